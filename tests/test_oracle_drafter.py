"""Pins for the oracle's drafter forward (Sec. 2.3, App. A.1) -- CPU only.

Checks against torch's fp64 library routines (scaled_dot_product_attention,
rms_norm, linear), the complex-number form of the rotary embedding, and an
explicit-loop brute force of a whole draft pass on a micro shape.
"""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as Fn

import oracle
from oracle import drafter as od
from paper_2609_37029_gb300 import synth

MICRO = synth.LspShape("micro", C=2, B=4, L=3, D=2, H=16, nq=4, nkv=2, d=8, F=24, V=40,
                       W=6, R=3, rc=5, dtype="f32", rope_theta=10000.0)


def _rng(seed):
    return np.random.default_rng(seed)


def test_context_attention_without_window_and_summary_is_block_self_attention():
    """W = R = 0: one bidirectional softmax over the block (torch SDPA, no mask, GQA)."""
    r = _rng(1)
    B, nq, nkv, d = 5, 6, 2, 8
    q, kb, vb = r.standard_normal((B, nq, d)), r.standard_normal((B, nkv, d)), r.standard_normal((B, nkv, d))
    empty = np.zeros((0, nkv, d))
    out = od.context_attention(q, kb, vb, empty, empty, np.zeros((nq, 0, d)), np.zeros((nq, 0, d)), d)
    tq = torch.from_numpy(q).permute(1, 0, 2)
    tk = torch.from_numpy(kb).permute(1, 0, 2).repeat_interleave(nq // nkv, dim=0)
    tv = torch.from_numpy(vb).permute(1, 0, 2).repeat_interleave(nq // nkv, dim=0)
    ref = Fn.scaled_dot_product_attention(tq, tk, tv).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(out, ref, atol=1e-13)


def test_context_attention_is_one_softmax_over_three_sources():
    """Eq. draft-context: [K^b; K^w; G] / [V^b; V^w; M] under a single normalisation."""
    r = _rng(2)
    B, nq, nkv, d, nw, R = 4, 4, 2, 8, 7, 3
    q = r.standard_normal((B, nq, d))
    kb, vb = r.standard_normal((B, nkv, d)), r.standard_normal((B, nkv, d))
    kw, vw = r.standard_normal((nw, nkv, d)), r.standard_normal((nw, nkv, d))
    G, M = r.standard_normal((nq, R, d)), r.standard_normal((nq, R, d))
    out = od.context_attention(q, kb, vb, kw, vw, G, M, d)
    rep = nq // nkv
    K = torch.cat([torch.from_numpy(kb).permute(1, 0, 2).repeat_interleave(rep, 0),
                   torch.from_numpy(kw).permute(1, 0, 2).repeat_interleave(rep, 0),
                   torch.from_numpy(G)], dim=1)
    V = torch.cat([torch.from_numpy(vb).permute(1, 0, 2).repeat_interleave(rep, 0),
                   torch.from_numpy(vw).permute(1, 0, 2).repeat_interleave(rep, 0),
                   torch.from_numpy(M)], dim=1)
    ref = Fn.scaled_dot_product_attention(torch.from_numpy(q).permute(1, 0, 2), K, V)
    np.testing.assert_allclose(out, ref.permute(1, 0, 2).numpy(), atol=1e-13)
    # the window is a set: any order of its rows gives the same result
    perm = r.permutation(nw)
    out2 = od.context_attention(q, kb, vb, kw[perm], vw[perm], G, M, d)
    np.testing.assert_allclose(out, out2, atol=1e-13)


def test_rope_matches_complex_rotation():
    r = _rng(3)
    x = r.standard_normal((6, 3, 16))
    pos = np.array([0, 1, 7, 4095, 65536, 131087])
    out = od.rope(x, pos, 1.0e6)
    half = 8
    inv = 1.0e6 ** (-np.arange(half) * 2.0 / 16)
    zc = (x[..., :half] + 1j * x[..., half:]) * np.exp(1j * pos[:, None, None] * inv[None, None, :])
    np.testing.assert_allclose(out[..., :half], zc.real, atol=1e-12)
    np.testing.assert_allclose(out[..., half:], zc.imag, atol=1e-12)
    # rotations preserve norms and make q.k depend only on the offset
    np.testing.assert_allclose(np.linalg.norm(out, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    q, k = r.standard_normal((1, 1, 16)), r.standard_normal((1, 1, 16))
    a = (od.rope(q, [10], 1e6) * od.rope(k, [3], 1e6)).sum()
    b = (od.rope(q, [1007], 1e6) * od.rope(k, [1000], 1e6)).sum()
    assert abs(a - b) < 1e-10


def test_rmsnorm_matches_torch():
    r = _rng(4)
    x, w = r.standard_normal((5, 32)) * 3, r.standard_normal(32)
    ref = Fn.rms_norm(torch.from_numpy(x), (32,), torch.from_numpy(w), eps=1e-6).numpy()
    np.testing.assert_allclose(od.rmsnorm(x, w, 1e-6), ref, atol=1e-13)


def _np_weights(shape, seed=5):
    w = synth.make_weights(shape, seed=seed)
    conv = lambda t: t.float().numpy()
    out = {k: conv(v) for k, v in w.items() if k != "layers"}
    out["layers"] = [{k: conv(v) for k, v in lw.items()} for lw in w["layers"]]
    return out


def _state(cfg, t, seed):
    r = _rng(seed)
    st = oracle.state_init(cfg)
    k = r.standard_normal((cfg.C, cfg.L, t, cfg.nkv, cfg.d))
    v = r.standard_normal((cfg.C, cfg.L, t, cfg.nkv, cfg.d))
    h = r.standard_normal((cfg.C, cfg.L, t, cfg.H))
    G = r.standard_normal((cfg.L, cfg.nq, cfg.R, cfg.d)) / math.sqrt(cfg.d)
    oracle.view_update(cfg, st, G, k, v, h, np.full(cfg.C, t))
    return st, G


def _brute_draft(cfg, st, w, toks, b):
    """Explicit loops, one scalar at a time, for one request (micro sizes only)."""
    def lin(W, x):  # y[n] = sum_k W[n][k] x[k]
        return [sum(W[n][kk] * x[kk] for kk in range(len(x))) for n in range(len(W))]

    def norm(x, wt):
        ms = sum(xi * xi for xi in x) / len(x)
        return [xi / math.sqrt(ms + cfg.rms_eps) * wi for xi, wi in zip(x, wt)]

    def rot(x, p):
        half = len(x) // 2
        out = list(x)
        for i in range(half):
            a = p * cfg.rope_theta ** (-2.0 * i / len(x))
            out[i] = x[i] * math.cos(a) - x[i + half] * math.sin(a)
            out[i + half] = x[i + half] * math.cos(a) + x[i] * math.sin(a)
        return out

    hcat = [st.hb[b][l][i] for l in range(cfg.L) for i in range(cfg.H)]
    c = lin(w["fuse"], hcat)
    x = []
    for i in range(cfg.B):
        e = w["embed"][toks[b][i]] if toks[b][i] >= 0 else w["mask_emb"]
        x.append([e[n] + w["pos"][i][n] + c[n] for n in range(cfg.H)])
    rep = cfg.nq // cfg.nkv
    for j in range(cfg.D):
        l = cfg.layer_map[j]
        lw = w["layers"][j]
        xn = [norm(xi, lw["in_norm"]) for xi in x]
        q = [[rot(norm(lin(lw["wq"], xi)[hh * cfg.d:(hh + 1) * cfg.d], lw["q_norm"]), st.t[b] + i)
              for hh in range(cfg.nq)] for i, xi in enumerate(xn)]
        k = [[rot(norm(lin(lw["wk"], xi)[g * cfg.d:(g + 1) * cfg.d], lw["k_norm"]), st.t[b] + i)
              for g in range(cfg.nkv)] for i, xi in enumerate(xn)]
        v = [[lin(lw["wv"], xi)[g * cfg.d:(g + 1) * cfg.d] for g in range(cfg.nkv)] for xi in xn]
        o = []
        for i in range(cfg.B):
            row = []
            for hh in range(cfg.nq):
                g = hh // rep
                keys = [k[jj][g] for jj in range(cfg.B)] + [list(r_[g]) for r_ in st.win_k[b][l]] \
                    + [list(gg) for gg in st_G[l][hh]]
                vals = [v[jj][g] for jj in range(cfg.B)] + [list(r_[g]) for r_ in st.win_v[b][l]] \
                    + [list(mm) for mm in st.m[b][l][hh]]
                s = [sum(q[i][hh][e] * kk[e] for e in range(cfg.d)) / math.sqrt(cfg.d) for kk in keys]
                mx = max(s)
                p = [math.exp(si - mx) for si in s]
                z = sum(p)
                row += [sum(p[n] * vals[n][e] for n in range(len(vals))) / z for e in range(cfg.d)]
            o.append(row)
        x = [[xi[n] + yo for n, yo in enumerate(lin(lw["wo"], oi))] for xi, oi in zip(x, o)]
        xn = [norm(xi, lw["post_norm"]) for xi in x]
        new = []
        for xi, xni in zip(x, xn):
            gt, up = lin(lw["w_gate"], xni), lin(lw["w_up"], xni)
            a = [gg / (1 + math.exp(-gg)) * uu for gg, uu in zip(gt, up)]
            new.append([xi[n] + yd for n, yd in enumerate(lin(lw["w_down"], a))])
        x = new
    return [lin(w["lm_head"], norm(xi, w["final_norm"])) for xi in x]


st_G = None


def test_draft_matches_explicit_loop_brute_force():
    global st_G
    cfg = MICRO
    st, G = _state(cfg, 9, 6)
    st_G = G
    w = _np_weights(cfg)
    w["G"] = G
    ow = oracle.OracleWeights(w)
    toks = np.array([[3, -1, -1, -1], [17, -1, 5, -1]])
    z0 = oracle.draft_base_logits(cfg, st, ow, toks)
    for b in range(cfg.C):
        w64 = {k: (np.asarray(v, np.float64) if k != "layers" else
                   [{kk: np.asarray(vv, np.float64) for kk, vv in lw.items()} for lw in v])
               for k, v in w.items()}
        ref = np.array(_brute_draft(cfg, st, w64, toks, b))
        np.testing.assert_allclose(z0[b], ref, rtol=1e-11, atol=1e-12)


TORCH_CFG = MICRO.with_(H=32, d=16, nq=4, nkv=2, F=48, V=64, W=8, R=4, D=3, L=2)


@pytest.mark.parametrize("variant", [
    {},                                  # the full drafter
    {"B": 7},                            # the paper's block size (7 drafts per round)
    {"W": 0},                            # ablation: w/o recent KV window (Sec. 3.4)
    {"R": 0},                            # ablation: w/o global summary
    {"no_boundary": True},               # ablation: w/o boundary state
    {"W": 0, "R": 0, "no_boundary": True},
])
def test_draft_matches_torch_composition(variant):
    """The same pass assembled from torch fp64 library calls (linear, rms_norm, SDPA, silu),
    for the full drafter and each variant of the ablation (a removed source is simply absent
    from the concatenated keys and values; without the boundary state the input slots carry
    no c_t)."""
    cfg = TORCH_CFG.with_(**variant)
    st, G = _state(cfg, 13, 7)
    w = _np_weights(cfg, seed=8)
    w["G"] = G
    toks = np.array([[1] + [-1] * (cfg.B - 2) + [2], [63] + [-1] * (cfg.B - 1)])
    z0 = oracle.draft_base_logits(cfg, st, oracle.OracleWeights(w), toks)
    T = lambda a: torch.from_numpy(np.asarray(a, dtype=np.float64))
    rep = cfg.nq // cfg.nkv
    for b in range(cfg.C):
        emb = torch.stack([T(w["embed"][t]) if t >= 0 else T(w["mask_emb"]) for t in toks[b]])
        x = emb + T(w["pos"])
        if not cfg.no_boundary:
            x = x + Fn.linear(T(st.hb[b]).reshape(-1), T(w["fuse"]))
        pos = torch.arange(cfg.B, dtype=torch.float64) + float(st.t[b])
        inv = cfg.rope_theta ** (-torch.arange(0, cfg.d, 2, dtype=torch.float64) / cfg.d)
        ang = pos[:, None] * inv[None, :]
        cos, sin = torch.cat([ang.cos()] * 2, -1)[:, None], torch.cat([ang.sin()] * 2, -1)[:, None]
        rot = lambda y: y * cos + torch.cat([-y[..., cfg.d // 2:], y[..., :cfg.d // 2]], -1) * sin
        for j in range(cfg.D):
            lw = {k: T(v) for k, v in w["layers"][j].items()}
            l = cfg.layer_map[j]
            xn = Fn.rms_norm(x, (cfg.H,), lw["in_norm"], cfg.rms_eps)
            q = Fn.rms_norm(Fn.linear(xn, lw["wq"]).view(cfg.B, cfg.nq, cfg.d), (cfg.d,), lw["q_norm"], cfg.rms_eps)
            k = Fn.rms_norm(Fn.linear(xn, lw["wk"]).view(cfg.B, cfg.nkv, cfg.d), (cfg.d,), lw["k_norm"], cfg.rms_eps)
            v = Fn.linear(xn, lw["wv"]).view(cfg.B, cfg.nkv, cfg.d)
            q, k = rot(q), rot(k)
            K = torch.cat([k.permute(1, 0, 2).repeat_interleave(rep, 0),
                           T(st.win_k[b][l]).permute(1, 0, 2).repeat_interleave(rep, 0), T(G[l])], 1)
            V = torch.cat([v.permute(1, 0, 2).repeat_interleave(rep, 0),
                           T(st.win_v[b][l]).permute(1, 0, 2).repeat_interleave(rep, 0), T(st.m[b, l])], 1)
            o = Fn.scaled_dot_product_attention(q.permute(1, 0, 2), K, V).permute(1, 0, 2).reshape(cfg.B, -1)
            x = x + Fn.linear(o, lw["wo"])
            xn = Fn.rms_norm(x, (cfg.H,), lw["post_norm"], cfg.rms_eps)
            x = x + Fn.linear(Fn.silu(Fn.linear(xn, lw["w_gate"])) * Fn.linear(xn, lw["w_up"]), lw["w_down"])
        ref = Fn.linear(Fn.rms_norm(x, (cfg.H,), T(w["final_norm"]), cfg.rms_eps), T(w["lm_head"]))
        np.testing.assert_allclose(z0[b], ref.numpy(), rtol=1e-11, atol=1e-12)


def test_without_boundary_equals_a_zero_fusion_matrix():
    """The no-boundary variant is the full drafter with W_fuse = 0, whatever h holds."""
    cfg = TORCH_CFG
    st, G = _state(cfg, 11, 12)
    w = _np_weights(cfg, seed=13)
    w["G"] = G
    toks = np.array([[5, -1, -1, -1], [9, -1, 4, -1]])
    z_nb = oracle.draft_base_logits(cfg.with_(no_boundary=True), st, oracle.OracleWeights(w), toks)
    w0 = dict(w, fuse=np.zeros_like(w["fuse"]))
    z_0 = oracle.draft_base_logits(cfg, st, oracle.OracleWeights(w0), toks)
    np.testing.assert_allclose(z_nb, z_0, rtol=1e-13, atol=1e-13)
    # and the boundary does matter for the full drafter
    assert np.abs(oracle.draft_base_logits(cfg, st, oracle.OracleWeights(w), toks) - z_0).max() > 1e-3


def test_state_bytes_of_the_ablation_variants():
    """Each removed source removes exactly its bytes from the per-request interface."""
    s = synth.Q8B
    full = oracle.state_bytes_per_request(s)
    assert full - oracle.state_bytes_per_request(s.with_(W=0)) == s.L * s.W * 2 * s.nkv * s.d * 2
    assert full - oracle.state_bytes_per_request(s.with_(R=0)) == s.L * s.nq * s.R * (s.d + 1) * 4
    assert full - oracle.state_bytes_per_request(s.with_(no_boundary=True)) == s.L * s.H * 2


def test_layer_pairing_reads_its_tapped_layer():
    """Changing the window of a tapped layer no draft layer reads leaves the logits unchanged."""
    cfg = MICRO.with_(L=3, D=1)          # l(0) = 0: layers 1 and 2 only feed the boundary
    st, G = _state(cfg, 9, 9)
    w = _np_weights(cfg, seed=10)
    w["G"] = G
    ow = oracle.OracleWeights(w)
    toks = np.array([[3, -1, -1, -1], [7, -1, -1, -1]])
    z_a = oracle.draft_base_logits(cfg, st, ow, toks)
    st.win_k[0][2] = st.win_k[0][2] + 1.0
    st.m[0, 1] += 1.0
    np.testing.assert_array_equal(z_a, oracle.draft_base_logits(cfg, st, ow, toks))
    st.win_k[0][0] = st.win_k[0][0] + 1.0
    assert not np.allclose(z_a[0], oracle.draft_base_logits(cfg, st, ow, toks)[0])
