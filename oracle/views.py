"""Fixed-size context interface (oracle side, fp64).  Test infrastructure only.

Restates Sec. 2.2 ("Fixed-Cost Context Interface"), Eq. global-summary, and the
incremental summary merge of App. A.2 (Eq. summary-update), plus the round
bookkeeping of Sec. 2.4 ("Inference"): after a verification that accepts r
candidates, the r+1 new KV rows (the committed token a and y_1..y_r) update the
summary and advance the recent window, and the hidden states of the last new row
give the new boundary.

State per request b (all float64 here):
  m[b][l][h][r][:]  summary value of query r of head h at tapped layer l
  eta[b][l][h][r]   its log-normaliser (-inf while no row has been folded)
  win_k[b][l], win_v[b][l]  the last <= W target K/V rows, oldest first, [n][nkv][d]
  hb[b][l][:]       target hidden state of the last folded row (boundary)
  t[b]              number of rows folded so far

Readings where the paper is silent: summary banks are per *query* head (the
paper's "each selected layer and attention head"), each scoring the key/value
head its query head shares under grouped-query attention (h // (nq/nkv)); the
summary queries G are used as given (no norm, no rotary embedding).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass
class OracleState:
    m: np.ndarray
    eta: np.ndarray
    win_k: list
    win_v: list
    hb: np.ndarray
    t: np.ndarray


def state_init(cfg) -> OracleState:
    """Empty interface: m = 0, eta = -inf, empty window, zero boundary, t = 0."""
    C, L, nq, R, d, nkv, H = cfg.C, cfg.L, cfg.nq, cfg.R, cfg.d, cfg.nkv, cfg.H
    return OracleState(
        m=np.zeros((C, L, nq, R, d)),
        eta=np.full((C, L, nq, R), -np.inf),
        win_k=[[np.zeros((0, nkv, d)) for _ in range(L)] for _ in range(C)],
        win_v=[[np.zeros((0, nkv, d)) for _ in range(L)] for _ in range(C)],
        hb=np.zeros((C, L, H)),
        t=np.zeros(C, dtype=np.int64),
    )


def _log_sum_exp(s):
    """log sum_j exp(s_j) along the last axis, evaluated with max subtraction (App. A.2)."""
    mx = np.max(s, axis=-1)
    return mx + np.log(np.sum(np.exp(s - mx[..., None]), axis=-1))


def summary_stats(g, K, V, d):
    """(eta_N, m_N) of App. A.2 for queries g [R][d] over a nonempty row set K, V [n][d].

    s_j = g^T k_j / sqrt(d);  eta_N = log sum_j exp(s_j);
    m_N = sum_j exp(s_j - eta_N) v_j.
    """
    s = g @ K.T / np.sqrt(d)                 # [R][n]
    eta_n = _log_sum_exp(s)                  # [R]
    m_n = np.exp(s - eta_n[:, None]) @ V     # [R][d]
    return eta_n, m_n


def merge(eta_a, m_a, eta_n, m_n):
    """Eq. summary-update: eta = log(e^eta_A + e^eta_N), m = e^(eta_A-eta) m_A + e^(eta_N-eta) m_N.

    Evaluated with max subtraction; eta_A = -inf (nothing folded yet) yields (eta_N, m_N).
    """
    mx = np.maximum(eta_a, eta_n)
    eta = mx + np.log(np.exp(eta_a - mx) + np.exp(eta_n - mx))
    m = np.exp(eta_a - eta)[:, None] * m_a + np.exp(eta_n - eta)[:, None] * m_n
    return eta, m


def view_update(cfg, st: OracleState, G, k_new, v_new, h_new, accepted_len):
    """Fold the newly accepted rows of one verification pass into the interface.

    G: [L][nq][R][d]; k_new, v_new: [C][L][>=n][nkv][d]; h_new: [C][L][>=n][H];
    accepted_len: [C] (n = accepted_len[b] rows per request; 0 leaves it unchanged).
    """
    G = np.asarray(G, dtype=np.float64)
    rep = cfg.nq // cfg.nkv
    for b in range(cfg.C):
        n = int(accepted_len[b])
        if n == 0:
            continue            # an empty new set leaves the state unchanged (App. A.2)
        for l in range(cfg.L):
            K = np.asarray(k_new[b, l, :n], dtype=np.float64)    # [n][nkv][d]
            V = np.asarray(v_new[b, l, :n], dtype=np.float64)
            for h in range(cfg.nq):
                g = h // rep
                eta_n, m_n = summary_stats(G[l, h], K[:, g], V[:, g], cfg.d)
                st.eta[b, l, h], st.m[b, l, h] = merge(st.eta[b, l, h], st.m[b, l, h], eta_n, m_n)
            # recent window: keep the last W rows (Sec. 2.2)
            st.win_k[b][l] = np.concatenate([st.win_k[b][l], K], axis=0)[-cfg.W:] if cfg.W > 0 else st.win_k[b][l][:0]
            st.win_v[b][l] = np.concatenate([st.win_v[b][l], V], axis=0)[-cfg.W:] if cfg.W > 0 else st.win_v[b][l][:0]
            # boundary: hidden state of the newest row at each tapped layer
            st.hb[b, l] = np.asarray(h_new[b, l, n - 1], dtype=np.float64)
        st.t[b] += n
    return st


def full_summary(G_lh, K, V, d):
    """Eq. global-summary recomputed from all rows: M_t = Attn(G, K_{1:t}, V_{1:t})."""
    s = G_lh @ K.T / np.sqrt(d)
    s = s - s.max(axis=1, keepdims=True)
    p = np.exp(s)
    p /= p.sum(axis=1, keepdims=True)
    return p @ V


def state_bytes_per_request(cfg, elem_bytes=2):
    """Persistent interface bytes per request in the stored layout.

    window K and V in the storage dtype: L * W * 2 * nkv * d elements;
    summary (m, eta) in fp32: L * nq * R * (d + 1) floats ("one value vector and
    one log-normalizer per query", App. A.2); boundary h: L * H elements
    (none in the ablation variant without the boundary state, Sec. 3.4).
    Independent of t (Sec. 2.4, "Fixed-cost complexity").
    """
    win = cfg.L * cfg.W * 2 * cfg.nkv * cfg.d * elem_bytes
    summ = cfg.L * cfg.nq * cfg.R * (cfg.d + 1) * 4
    bnd = 0 if getattr(cfg, "no_boundary", False) else cfg.L * cfg.H * elem_bytes
    return win + summ + bnd
