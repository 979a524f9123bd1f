"""Prefill (Sec. 2.2, Eq. global-summary, App. A.2, Fig. 3): the summary of a
whole prefix built in one call, checked against the oracle's fold of the same
rows into an empty request (the summary of all rows at once)."""
import numpy as np
import pytest
import torch

import oracle
from tests.gpu_common import check_view_state, export_state, f64, fold_chunk, lsp_lib
from paper_2609_37029_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lsp():
    return lsp_lib()


PF = synth.LspShape("pf", C=3, B=16, L=2, D=1, H=256, nq=8, nkv=2, d=128, F=256, V=1024, W=40,
                    R=16, rc=16)


def _prefill_both(lsp, st, ost, s, b, t, seed, Gn):
    """Request b's whole prefix of t rows: lsp_prefill on the GPU, an empty-state fold in the oracle."""
    k, v, h = synth.make_features(s, t, seed=seed)
    lsp.lsp_prefill(st, b, k[b].contiguous().cuda(), v[b].contiguous().cuda(), h[b].contiguous().cuda())
    acc = np.zeros(s.C, dtype=np.int32)
    acc[b] = t
    # the oracle request starts empty (the prefill replaces it)
    fresh = oracle.state_init(s.with_(C=1))
    oracle.view_update(s.with_(C=1), fresh, Gn, f64(k[b:b + 1]), f64(v[b:b + 1]), f64(h[b:b + 1]),
                       acc[b:b + 1])
    ost.eta[b], ost.m[b], ost.hb[b], ost.t[b] = fresh.eta[0], fresh.m[0], fresh.hb[0], fresh.t[0]
    ost.win_k[b], ost.win_v[b] = fresh.win_k[0], fresh.win_v[0]


@pytest.mark.parametrize("t", [1, 37, 64, 65, 300, 4096, 5000])
def test_prefill_matches_oracle(lsp, t):
    s = PF
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        w = synth.make_weights(s, seed=3)
        lsp.lsp_state_init(st, w["G"].cuda())
        ost = oracle.state_init(s)
        Gn = f64(w["G"])
        _prefill_both(lsp, st, ost, s, 1, t, 200 + t, Gn)
        torch.cuda.synchronize()
        check_view_state(lsp, st, ost, s)        # requests 0 and 2 stay empty on both sides
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


@pytest.mark.parametrize("variant", [{"R": 0}, {"W": 0}, {"no_boundary": True}])
def test_prefill_ablation_variants(lsp, variant):
    """Without the summary (R = 0) only the window, boundary and t are written; without the
    window (W = 0) only the summary; without the boundary no hidden state is read (h = None)."""
    s = PF.with_(**variant)
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        w = synth.make_weights(s, seed=3)
        lsp.lsp_state_init(st, w["G"].cuda() if w["G"].numel() else None)
        ost = oracle.state_init(s)
        Gn = f64(w["G"])
        t = 777
        k, v, h = synth.make_features(s, t, seed=55)
        hb = None if s.no_boundary else h[1].contiguous().cuda()
        lsp.lsp_prefill(st, 1, k[1].contiguous().cuda(), v[1].contiguous().cuda(), hb)
        fresh = oracle.state_init(s.with_(C=1))
        oracle.view_update(s.with_(C=1), fresh, Gn, f64(k[1:2]), f64(v[1:2]), f64(h[1:2]),
                           np.array([t], dtype=np.int32))
        ost.eta[1], ost.m[1], ost.hb[1], ost.t[1] = fresh.eta[0], fresh.m[0], fresh.hb[0], fresh.t[0]
        ost.win_k[1], ost.win_v[1] = fresh.win_k[0], fresh.win_v[0]
        torch.cuda.synchronize()
        check_view_state(lsp, st, ost, s)
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


def test_prefill_replaces_state_and_rounds_continue(lsp):
    """A prefill overwrites a request that already holds rows; later view updates fold on top."""
    s = PF
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        w = synth.make_weights(s, seed=4)
        lsp.lsp_state_init(st, w["G"].cuda())
        ost = oracle.state_init(s)
        Gn = f64(w["G"])
        k, v, h = synth.make_features(s, 50, seed=7)
        fold_chunk(lsp, st, ost, s, Gn, k, v, h, torch.tensor([50, 20, 3], dtype=torch.int32))
        for b, t in [(0, 777), (2, 130)]:
            _prefill_both(lsp, st, ost, s, b, t, 300 + b, Gn)
        for r, acc in enumerate([[5, 17, 1], [0, 9, 33]]):
            k, v, h = synth.make_features(s, 40, seed=400 + r)
            fold_chunk(lsp, st, ost, s, Gn, k, v, h, torch.tensor(acc, dtype=torch.int32))
        torch.cuda.synchronize()
        check_view_state(lsp, st, ost, s)
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


def test_prefill_equals_incremental_fold_on_gpu(lsp):
    """Eq. summary-update is exact: one prefill and a chunked fold agree (fp32 tolerance)."""
    s = PF
    sts = [lsp.lsp_state_create(lsp.make_config(s)) for _ in range(2)]
    try:
        w = synth.make_weights(s, seed=5)
        for st in sts:
            lsp.lsp_state_init(st, w["G"].cuda())
        t = 3000
        k, v, h = synth.make_features(s, t, seed=9)
        lsp.lsp_prefill(sts[0], 0, k[0].contiguous().cuda(), v[0].contiguous().cuda(), h[0].contiguous().cuda())
        for c0 in range(0, t, 700):
            n = min(700, t - c0)
            acc = torch.tensor([n, 0, 0], dtype=torch.int32).cuda()
            lsp.lsp_view_update(sts[1], k[:, :, c0:c0 + n].contiguous().cuda(),
                                v[:, :, c0:c0 + n].contiguous().cuda(), h[:, :, c0:c0 + n].contiguous().cuda(), acc)
        torch.cuda.synchronize()
        a, b = export_state(lsp, sts[0], s), export_state(lsp, sts[1], s)
        np.testing.assert_allclose(a["m"].double().numpy(), b["m"].double().numpy(), rtol=0, atol=5e-5)
        np.testing.assert_allclose(a["eta"].double().numpy(), b["eta"].double().numpy(), rtol=0, atol=5e-4)
        for key in ("win_k", "win_v", "h", "t"):
            assert torch.equal(a[key], b[key]), key
    finally:
        for st in sts:
            lsp.lsp_state_destroy(st)


def test_prefill_with_the_last_hidden_row_only(lsp):
    """h_rows = 1: h carries only the prefix's last row, the one the boundary reads."""
    s = PF
    sts = [lsp.lsp_state_create(lsp.make_config(s)) for _ in range(2)]
    try:
        G = synth.make_weights(s, seed=3)["G"].cuda()
        for st in sts:
            lsp.lsp_state_init(st, G)
        k, v, h = synth.make_features(s, 300, seed=77)
        kb, vb, hb = k[2].contiguous().cuda(), v[2].contiguous().cuda(), h[2].contiguous().cuda()
        lsp.lsp_prefill(sts[0], 2, kb, vb, hb)
        lsp.lsp_prefill(sts[1], 2, kb, vb, hb[:, -1:].contiguous(), h_rows=1)
        torch.cuda.synchronize()
        ea, eb = export_state(lsp, sts[0], s), export_state(lsp, sts[1], s)
        for key in ea:
            assert torch.equal(ea[key], eb[key]), key
    finally:
        for st in sts:
            lsp.lsp_state_destroy(st)


@pytest.mark.slow
def test_prefill_128k_at_qwen3_8b_heads_sampled(lsp):
    """128K rows at the Qwen3-8B head shape (32 q / 8 kv x 128, R = 16), one tapped layer:
    sampled query heads against the oracle's summary statistics in fp64."""
    s = synth.Q8B.with_(C=1, L=1, D=1, V=1024, F=256)
    t = 131072
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        w = synth.make_weights(s, seed=6)
        lsp.lsp_state_init(st, w["G"].cuda())
        k, v, h = synth.make_features(s, t, seed=11, device="cuda")
        lsp.lsp_prefill(st, 0, k[0], v[0], h[0])
        torch.cuda.synchronize()
        ex = export_state(lsp, st, s)
        assert int(ex["t"][0]) == t
        G = f64(w["G"])
        rep = s.nq // s.nkv
        for hq in [0, 5, 17, 31]:
            g = hq // rep
            K = f64(k[0, 0, :, g])
            V = f64(v[0, 0, :, g])
            eta_o, m_o = oracle.views.summary_stats(G[0, hq], K, V, s.d)
            np.testing.assert_allclose(ex["m"][0, 0, hq].double().numpy(), m_o, rtol=0, atol=1e-4)
            np.testing.assert_allclose(ex["eta"][0, 0, hq].double().numpy(), eta_o, rtol=0, atol=1e-3)
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


def test_prefill_rejects_unsupported_and_bad_args(lsp):
    s32 = PF.with_(dtype="f32", nq=4, d=64)
    st = lsp.lsp_state_create(lsp.make_config(s32))
    try:
        w = synth.make_weights(s32, seed=3)
        lsp.lsp_state_init(st, w["G"].cuda())
        k, v, h = synth.make_features(s32, 10, seed=1)
        with pytest.raises(lsp.LspError) as e:
            lsp.lsp_prefill(st, 0, k[0].contiguous().cuda(), v[0].contiguous().cuda(), h[0].contiguous().cuda())
        assert e.value.status == lsp.LSP_ERR_UNSUPPORTED
    finally:
        lsp.lsp_state_destroy(st)
    st = lsp.lsp_state_create(lsp.make_config(PF))
    try:
        w = synth.make_weights(PF, seed=3)
        lsp.lsp_state_init(st, w["G"].cuda())
        k, v, h = synth.make_features(PF, 10, seed=1)
        with pytest.raises(lsp.LspError) as e:
            lsp.lsp_prefill(st, PF.C, k[0].contiguous().cuda(), v[0].contiguous().cuda(), h[0].contiguous().cuda())
        assert e.value.status == lsp.LSP_ERR_ARG
    finally:
        lsp.lsp_state_destroy(st)
