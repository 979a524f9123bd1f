"""Markov correction and sequential proposal sampling (oracle side, fp64).  Test infrastructure only.

Restates Eq. markov and Eq. proposal-factorization (Sec. 2.3): with y_0 = a,
    z_i = z_i^(0) + W_c E_c(y_{i-1}),   q_i = softmax(z_i),   y_i ~ q_i,
for i = 1..B in order; the corrected z_i are the distributions verification uses.

Readings where the paper is silent:
* E_c is a [V][r_c] table (row y is E_c(y)); W_c is [V][r_c], so W_c E_c(y) is
  the length-V vector W_c @ E_c[y].
* Sampling at temperature T > 0 is Gumbel-max: y = argmax_v (z_v / T + g_v) with
  g_v = -log(-log u_v), u_v = ((x_v >> 9) + 1/2) * 2^-23 and x_v the Philox word
  of (request b, step i, round, v).  T = 0 is greedy: y = argmax_v z_v.
* Ties go to the lowest vocabulary index.  The argmax decision is taken on the
  score rounded to fp32: the paper fixes no precision for it, so the oracle
  decides in the CUDA sampler's.  Positions are compared only where the fp64
  top-1/top-2 margin exceeds 1e-2, where an fp64 argmax would agree.
"""
from __future__ import annotations

import numpy as np

from .philox import sampler_words


def gumbel(seed, rnd, b, i, V):
    """Gumbel(0, 1) noise for every vocabulary entry at (b, i, round), fp64 [V]."""
    x = sampler_words(seed, rnd, b, i, V)
    u = ((x >> np.uint32(9)).astype(np.float64) + 0.5) * 2.0 ** -23
    return -np.log(-np.log(u))


def _top2_margin(score):
    if score.shape[0] < 2:
        return np.inf
    top = np.partition(score, -2)[-2:]
    return float(top[1] - top[0])


def sample_block(z0_b, a, Ec, Wc, temperature, seed, rnd, b, forced_prev=None):
    """Sequential correction + sampling for one request.

    z0_b: [B][V] base logits; a: committed token (y_0); Ec, Wc: [V][rc].
    forced_prev: optional [B] tokens; when given, step i >= 1 conditions on
    forced_prev[i-1] instead of its own y_{i-1} (teacher forcing, used to keep
    later steps comparable after a token mismatch).
    Returns (tokens [B] int64, corrected logits [B][V] fp64, margins [B] fp64).
    """
    z0_b = np.asarray(z0_b, dtype=np.float64)
    Ec = np.asarray(Ec, dtype=np.float64)
    Wc = np.asarray(Wc, dtype=np.float64)
    B, V = z0_b.shape
    toks = np.zeros(B, dtype=np.int64)
    zs = np.zeros((B, V))
    margins = np.zeros(B)
    y_prev = int(a)
    for i in range(B):
        z = z0_b[i] + Wc @ Ec[y_prev]
        if temperature > 0:
            score = z / temperature + gumbel(seed, rnd, b, i, V)
        else:
            score = z
        y = int(np.argmax(score.astype(np.float32)))
        toks[i], zs[i], margins[i] = y, z, _top2_margin(score)
        y_prev = int(forced_prev[i]) if forced_prev is not None else y
    return toks, zs, margins
