"""Target-side verification of a drafted block (oracle side, fp64).  Test infrastructure only.

Restates the speculative-decoding rule of Sec. 2.1 (Preliminaries): the drafted
candidates y_1..y_B, drawn from q_i, are tested in order; y_i is accepted with
probability alpha_i = min(1, p_i(y_i) / q_i(y_i)) (Eq. acceptance).  At the
first rejected position i the rest of the block is discarded and a correction
token is drawn from p_i^corr(v) = [p_i(v) - q_i(v)]_+ / sum_u [p_i(u) - q_i(u)]_+
(Eq. residual).  If all B candidates are accepted, one more token is drawn from
p_{B+1} = p(. | s, y_{1:B}).  A round thus emits r + 1 tokens (r accepted).

Readings where the paper is silent:
* p_i = softmax(target logits_i / T) and q_i = softmax(draft logits_i / T) at the
  round's sampling temperature T; the draft logits are the sampler's corrected
  z_i (the distributions the candidates were drawn from).
* T = 0 is the greedy limit: y_i is accepted iff y_i = argmax_v p_i (lowest index
  on ties), and the emitted token after r accepted candidates is argmax p_{r+1}.
* Randomness is Philox4x32-10 with the drafting key (seed).  The acceptance
  uniform of position i is word 0 of counter (0, 2^30 + i, b, round), mapped
  u = ((x >> 9) + 1/2) 2^-23, and y_i is accepted iff u * q_i(y_i) < p_i(y_i)
  (u < alpha_i without a division).  The correction or bonus draw at position i
  is Gumbel-max over the words of counters (v >> 2, 2^31 + i, b, round):
  argmax_v (log w_v + g_v) with w = [p_i - q_i]_+ (correction) or w = p_{B+1}
  (bonus).  These counters never coincide with the drafter's (its second word
  is a step index < 2^30).
* Decisions are taken on fp32-rounded scores, the precision the CUDA kernels
  decide in; the returned margins tell a test how close each decision was.
"""
from __future__ import annotations

import numpy as np

from .philox import sampler_words

ACCEPT_STREAM = 1 << 30
DRAW_STREAM = 1 << 31


def _softmax(z):
    z = z - np.max(z)
    e = np.exp(z)
    return e / np.sum(e)


def accept_uniform(seed, rnd, b, i):
    """The acceptance uniform of position i of request b (fp64 in (0, 1))."""
    x = sampler_words(seed, rnd, b, ACCEPT_STREAM + i, 1)[0]
    return (float(x >> np.uint32(9)) + 0.5) * 2.0 ** -23


def draw_gumbel(seed, rnd, b, i, V):
    """Gumbel noise of the correction / bonus draw at position i, fp64 [V]."""
    x = sampler_words(seed, rnd, b, DRAW_STREAM + i, V)
    u = ((x >> np.uint32(9)).astype(np.float64) + 0.5) * 2.0 ** -23
    return -np.log(-np.log(u))


def _argmax_with_margin(score):
    s32 = score.astype(np.float32)
    k = int(np.argmax(s32))
    finite = np.sort(s32[np.isfinite(s32)])
    margin = float(finite[-1]) - float(finite[-2]) if finite.size > 1 else np.inf
    return k, margin


def verify_block(zt, zq, y, temperature, seed, rnd, b):
    """Verify one request's drafted block.

    zt: [B+1][V] target logits (position B is p(. | s, y_1..y_B));
    zq: [B][V] draft logits (the corrected z_i); y: [B] drafted tokens.
    Returns (r, token, accept_margins, draw_margin): r accepted candidates, the
    emitted correction / bonus token, |u q_i(y_i) - p_i(y_i)| / max(...) for each
    tested position, and the top-2 gap of the final draw's fp32 score.
    """
    zt = np.asarray(zt, dtype=np.float64)
    zq = np.asarray(zq, dtype=np.float64)
    B = zq.shape[0]
    V = zt.shape[1]
    margins = []
    if temperature <= 0:
        for i in range(B):
            k, m = _argmax_with_margin(zt[i])
            margins.append(m)
            if int(y[i]) != k:
                return i, k, margins, m
        k, m = _argmax_with_margin(zt[B])
        return B, k, margins, m
    for i in range(B):
        p = _softmax(zt[i] / temperature)
        q = _softmax(zq[i] / temperature)
        u = accept_uniform(seed, rnd, b, i)
        lhs, rhs = u * q[int(y[i])], p[int(y[i])]
        margins.append(abs(lhs - rhs) / max(lhs, rhs, 1e-300))
        if not lhs < rhs:
            w = np.maximum(p - q, 0.0)
            with np.errstate(divide="ignore"):
                score = np.log(w) + draw_gumbel(seed, rnd, b, i, V)
            k, m = _argmax_with_margin(score)
            return i, k, margins, m
    p = _softmax(zt[B] / temperature)
    with np.errstate(divide="ignore"):
        score = np.log(p) + draw_gumbel(seed, rnd, b, B, V)
    k, m = _argmax_with_margin(score)
    return B, k, margins, m
