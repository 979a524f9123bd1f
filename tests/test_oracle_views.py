"""Pins for the oracle's context interface (Sec. 2.2, App. A.2) -- CPU only.

Each check ties the oracle to something other than itself: the full-prefix
attention of Eq. global-summary evaluated by torch's fp64 attention routine,
closed forms (G = 0 gives the mean of V), the paper's printed state sizes, and
brute-force slices of the prefix.
"""
import os

import numpy as np
import pytest
import torch
from scipy.special import logsumexp

import oracle
from paper_2609_37029_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")

MICRO = synth.LspShape("micro", C=3, B=4, L=2, D=2, H=16, nq=4, nkv=2, d=8, F=24, V=40,
                       W=6, R=3, rc=5, dtype="f32")


def _prefix(cfg, t, seed):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((cfg.C, cfg.L, t, cfg.nkv, cfg.d))
    v = rng.standard_normal((cfg.C, cfg.L, t, cfg.nkv, cfg.d))
    h = rng.standard_normal((cfg.C, cfg.L, t, cfg.H))
    return k, v, h


def _queries(cfg, seed, scale=None):
    rng = np.random.default_rng(seed)
    s = (1.0 / cfg.d) ** 0.5 if scale is None else scale
    return rng.standard_normal((cfg.L, cfg.nq, cfg.R, cfg.d)) * s


def _fold(cfg, G, k, v, h, chunks):
    """Fold rows 0..t-1 chunk by chunk; `chunks` is a list of per-request chunk sizes."""
    st = oracle.state_init(cfg)
    pos = np.zeros(cfg.C, dtype=np.int64)
    for acc in chunks:
        acc = np.asarray(acc)
        kk = np.zeros((cfg.C, cfg.L, max(1, acc.max()), cfg.nkv, cfg.d))
        vv = np.zeros_like(kk)
        hh = np.zeros((cfg.C, cfg.L, max(1, acc.max()), cfg.H))
        for b in range(cfg.C):
            kk[b, :, :acc[b]] = k[b, :, pos[b]:pos[b] + acc[b]]
            vv[b, :, :acc[b]] = v[b, :, pos[b]:pos[b] + acc[b]]
            hh[b, :, :acc[b]] = h[b, :, pos[b]:pos[b] + acc[b]]
        oracle.view_update(cfg, st, G, kk, vv, hh, acc)
        pos += acc
    return st


def _sdpa_summary(G_lh, K, V):
    """Eq. global-summary via torch's fp64 attention (library routine)."""
    q = torch.from_numpy(G_lh)[None]
    out = torch.nn.functional.scaled_dot_product_attention(
        q, torch.from_numpy(K)[None], torch.from_numpy(V)[None])
    return out[0].numpy()


@pytest.mark.parametrize("chunk", [1, 3, 17, 50])
def test_incremental_merge_equals_full_attention(chunk):
    cfg, t = MICRO, 50
    k, v, h = _prefix(cfg, t, 1)
    G = _queries(cfg, 2)
    chunks = []
    left = t
    while left > 0:
        c = min(chunk, left)
        chunks.append([c] * cfg.C)
        left -= c
    st = _fold(cfg, G, k, v, h, chunks)
    rep = cfg.nq // cfg.nkv
    for b in range(cfg.C):
        for l in range(cfg.L):
            for hq in range(cfg.nq):
                g = hq // rep
                ref = _sdpa_summary(G[l, hq], k[b, l, :, g], v[b, l, :, g])
                np.testing.assert_allclose(st.m[b, l, hq], ref, rtol=0, atol=1e-12)
                s = G[l, hq] @ k[b, l, :, g].T / np.sqrt(cfg.d)
                np.testing.assert_allclose(st.eta[b, l, hq], logsumexp(s, axis=1), rtol=1e-13, atol=1e-12)
    assert list(st.t) == [t] * cfg.C


def test_ragged_chunks_per_request():
    """Different requests fold different chunk sequences; each matches its full prefix."""
    cfg, t = MICRO, 30
    k, v, h = _prefix(cfg, t, 3)
    G = _queries(cfg, 4)
    seqs = [[1, 5, 0, 24], [17, 13, 0, 0], [0, 0, 30, 0]]
    chunks = [[seqs[b][r] for b in range(cfg.C)] for r in range(4)]
    st = _fold(cfg, G, k, v, h, chunks)
    for b in range(cfg.C):
        ref = _sdpa_summary(G[1, 3], k[b, 1, :, 1], v[b, 1, :, 1])
        np.testing.assert_allclose(st.m[b, 1, 3], ref, atol=1e-12)


def test_empty_new_set_leaves_state_unchanged():
    cfg = MICRO
    k, v, h = _prefix(cfg, 10, 5)
    G = _queries(cfg, 6)
    st = _fold(cfg, G, k, v, h, [[4, 4, 4]])
    before = (st.m.copy(), st.eta.copy(), st.hb.copy(), st.t.copy(),
              [[w.copy() for w in ws] for ws in st.win_k])
    oracle.view_update(cfg, st, G, k[:, :, 4:], v[:, :, 4:], h[:, :, 4:], np.array([0, 0, 0]))
    assert np.array_equal(st.m, before[0]) and np.array_equal(st.eta, before[1])
    assert np.array_equal(st.hb, before[2]) and np.array_equal(st.t, before[3])
    for b in range(cfg.C):
        for l in range(cfg.L):
            assert np.array_equal(st.win_k[b][l], before[4][b][l])


def test_zero_queries_give_mean_of_values():
    cfg, t = MICRO, 23
    k, v, h = _prefix(cfg, t, 7)
    G = np.zeros((cfg.L, cfg.nq, cfg.R, cfg.d))
    st = _fold(cfg, G, k, v, h, [[5] * 3, [11] * 3, [7] * 3])
    rep = cfg.nq // cfg.nkv
    for hq in range(cfg.nq):
        mean = v[2, 0, :, hq // rep].mean(axis=0)
        for r in range(cfg.R):
            np.testing.assert_allclose(st.m[2, 0, hq, r], mean, atol=1e-13)
            assert abs(st.eta[2, 0, hq, r] - np.log(t)) < 1e-13


def test_large_scores_stay_finite():
    """Max subtraction (App. A.2): scores near 1e3 neither overflow nor lose the result."""
    cfg, t = MICRO, 40
    k, v, h = _prefix(cfg, t, 8)
    G = _queries(cfg, 9, scale=300.0)
    st = _fold(cfg, G, k, v, h, [[7] * 3] * 5 + [[5] * 3])
    assert np.isfinite(st.m).all() and np.isfinite(st.eta).all()
    ref = _sdpa_summary(G[0, 0], k[0, 0, :, 0], v[0, 0, :, 0])
    np.testing.assert_allclose(st.m[0, 0, 0], ref, atol=1e-10)


@pytest.mark.parametrize("t", [4, 6, 31])
def test_window_is_last_W_rows_and_boundary_is_last_row(t):
    cfg = MICRO
    k, v, h = _prefix(cfg, t, 10)
    G = _queries(cfg, 11)
    chunks, left = [], t
    while left > 0:
        c = min(4, left)
        chunks.append([c] * 3)
        left -= c
    st = _fold(cfg, G, k, v, h, chunks)
    lo = max(0, t - cfg.W)
    for b in range(cfg.C):
        for l in range(cfg.L):
            assert np.array_equal(st.win_k[b][l], k[b, l, lo:t])
            assert np.array_equal(st.win_v[b][l], v[b, l, lo:t])
            assert np.array_equal(st.hb[b, l], h[b, l, t - 1])


def _golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                key, val = line.split()
                vals[key] = float(val)
    return vals


def test_state_size_matches_paper_and_is_constant_in_t():
    """Sec. 3.3: ~6.3 MiB fixed drafter state vs DSpark 640 -> 2560 MiB; 406x at 128K."""
    g = _golden("state_size_qwen3_8b.txt")
    q8b = synth.Q8B
    per_req = oracle.state_bytes_per_request(q8b, elem_bytes=2) / 2 ** 20
    assert abs(per_req - g["longspark_state_mib"]) < 0.05
    # DSpark keeps every retained token's K and V at the 5 tapped layers (bf16).
    dspark = lambda t: t * q8b.L * 2 * q8b.nkv * q8b.d * 2 / 2 ** 20
    assert dspark(32768) == g["dspark_state_mib_32k"]
    assert dspark(131072) == g["dspark_state_mib_128k"]
    assert round(dspark(131072) / per_req) == g["reduction_128k"]
    # and the oracle's arrays do not grow with t
    cfg = MICRO
    G = _queries(cfg, 12)
    sizes = []
    for t in (3, 30, 90):
        k, v, h = _prefix(cfg, t, 13)
        st = _fold(cfg, G, k, v, h, [[t] * 3])
        sizes.append(st.m.nbytes + st.eta.nbytes + st.hb.nbytes
                     + sum(w.nbytes for ws in st.win_k for w in ws) * 2)
    assert sizes[1] == sizes[2]
