"""GPU parity of the individual kernels through the C ABI against the fp64 oracle.

* Philox words: bit-exact with the oracle's restatement.
* Projection GEMM (tcgen05, bf16 and tf32): vs an fp64 matmul of the same
  stored inputs, several tiles, ragged M / N / K, split-K on and off.
* View update (Eq. summary-update, window ring, boundary, t): vs the oracle
  after ragged chunk sequences including empty and larger-than-W updates.
* Correction + sampler (Eq. markov, Eq. proposal-factorization): tokens
  bit-exact wherever the oracle's top-1/top-2 margin exceeds 1e-2, corrected
  logits to fp32 accuracy, under teacher forcing.
"""
import math

import numpy as np
import pytest
import torch

import oracle
from oracle import philox
from paper_2609_37029_gb300 import synth
from tests.gpu_common import (check_view_state, export_state, f64, fold_chunk, lsp_lib)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lsp():
    return lsp_lib()


def test_philox_stream_matches_oracle(lsp):
    for seed, rnd, b, i, n in [(7, 0, 0, 0, 4096), (0xDEADBEEF12345678, 77, 15, 3, 1000),
                               (2 ** 64 - 1, 2 ** 32 - 1, 31, 15, 151936)]:
        out = torch.empty(n, dtype=torch.int32, device="cuda")
        lsp.lsp_philox_words(seed, rnd, b, i, out, n)
        got = out.cpu().numpy().view(np.uint32)
        want = philox.sampler_words(seed, rnd, b, i, n)
        assert np.array_equal(got, want)


LINEAR_CASES = [
    # M, N, K, dtype, splits
    (1, 128, 64, "bf16", 1),
    (16, 256, 320, "bf16", 1),
    (40, 384, 4096, "bf16", 3),
    (256, 1024, 4096, "bf16", 1),
    (256, 640, 1000, "bf16", 4),
    (300, 200, 136, "bf16", 1),
    (512, 256, 512, "bf16", 2),
    (256, 512, 4096, "bf16", 8),
    (16, 384, 20480, "bf16", 8),     # the boundary-fusion shape (M = C)
    (200, 256, 2048, "bf16", 4),     # ragged token count
    (96, 256, 1024, "bf16", 5),
    (256, 256, 1024, "bf16", 12),
    (256, 2560, 1024, "bf16", 8),    # >= 2 CTAs per SM
    (250, 19456, 512, "bf16", 1),    # ragged M, one split, 152 weight tiles
    (256, 40000, 512, "bf16", 1),    # >= 2 x SMs tiles, fp32 out: the persistent one-CTA-per-SM form
    (100, 40000, 256, "bf16", 1),    # the same with a ragged token count (112-token tile)
    (8, 128, 256, "f32", 1),
    (64, 384, 260, "f32", 3),
    (64, 384, 520, "f32", 2),
]


@pytest.mark.parametrize("M,N,K,dt,splits", LINEAR_CASES)
def test_linear_matches_fp64_matmul(lsp, M, N, K, dt, splits):
    """One split writes Y directly; more write fp32 partials that a sum kernel adds in
    split order."""
    g = torch.Generator().manual_seed(M * 7 + N + K)
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    X = torch.randn(M, K, generator=g).to(tdt)
    W = (torch.randn(N, K, generator=g) * 0.05).to(tdt)
    Y = torch.full((M, N), float("nan"), device="cuda")
    nbytes = lsp.lsp_linear_workspace_bytes(M, N, splits)
    ws = torch.zeros(max(nbytes, 4), dtype=torch.uint8, device="cuda")
    code = lsp.LSP_DTYPE_BF16 if dt == "bf16" else lsp.LSP_DTYPE_F32
    prev = None
    for _ in range(2):              # second call reuses the workspace (counters reset)
        lsp.lsp_linear(X.cuda(), W.cuda(), Y, M, N, K, code, splits, ws, nbytes)
        torch.cuda.synchronize()
        ref = f64(X) @ f64(W).T
        got = f64(Y)
        if prev is not None:        # split-K sums in a fixed order: bit-identical reruns
            assert np.array_equal(got, prev)
        prev = got.copy()
        scale = np.abs(ref).max()
        # bf16 operands are exact; tf32 rounds operands to 10 mantissa bits
        tol = 1e-5 if dt == "bf16" else 4e-3
        assert np.isfinite(got).all()
        assert np.abs(got - ref).max() <= tol * scale, np.abs(got - ref).max() / scale


VU = synth.LspShape("vu", C=3, B=16, L=2, D=1, H=256, nq=8, nkv=2, d=128, F=256, V=1024, W=40,
                    R=16, rc=16)
VU32 = VU.with_(name="vu32", dtype="f32", nq=4, d=64)
# rep * R summary queries per KV head: 64 above; the tensor-core kernel takes every
# multiple of 16 up to 128 (16 x 1..8), the FMA kernel the rest
VU_Q = {"q16": VU.with_(name="vu16", nq=2), "q48": VU.with_(name="vu48", nq=6),
        "q80": VU.with_(name="vu80", nq=10), "q128": VU.with_(name="vu128", nq=8, nkv=1),
        "q24-fma": VU.with_(name="vu24", R=6)}


@pytest.mark.parametrize("s", [VU, VU32, *VU_Q.values()], ids=["bf16", "f32", *VU_Q])
def test_view_update_matches_oracle(lsp, s):
    cfg = lsp.make_config(s)
    st = lsp.lsp_state_create(cfg)
    try:
        w = synth.make_weights(s, seed=3)
        G = w["G"]
        lsp.lsp_state_init(st, G.cuda())
        ost = oracle.state_init(s)
        Gn = f64(G)
        seqs = [[5, 1, 17], [0, 33, 2], [64, 0, 41], [1, 1, 0], [17, 17, 17], [40, 3, 80]]
        for r, acc in enumerate(seqs):
            rows = max(acc) + 2
            k, v, h = synth.make_features(s, rows, seed=100 + r)
            fold_chunk(lsp, st, ost, s, Gn, k, v, h, torch.tensor(acc, dtype=torch.int32))
        torch.cuda.synchronize()
        check_view_state(lsp, st, ost, s)
        rc, bits = lsp.lsp_get_error(st)
        assert rc == lsp.LSP_OK and bits == 0
    finally:
        lsp.lsp_state_destroy(st)


def test_boundary_row_only_features_match_full_rows(lsp):
    """h_rows = 1 (each request's boundary row only) gives the same state as the full rows,
    and h_rows values other than 0, 1 and rows are rejected."""
    s = VU
    cfg = lsp.make_config(s)
    a, b2 = lsp.lsp_state_create(cfg), lsp.lsp_state_create(cfg)
    try:
        G = synth.make_weights(s, seed=6)["G"].cuda()
        lsp.lsp_state_init(a, G)
        lsp.lsp_state_init(b2, G)
        for r, acc in enumerate([[5, 1, 17], [16, 3, 0], [2, 40, 9]]):
            rows = max(acc) + 2
            k, v, h = synth.make_features(s, rows, seed=300 + r, device="cuda")
            acc_t = torch.tensor(acc, dtype=torch.int32, device="cuda")
            # the boundary row of each (request, layer); requests with no new row keep row 0
            idx = (acc_t.long().clamp(min=1) - 1).view(s.C, 1, 1, 1).expand(s.C, s.L, 1, s.H)
            h_last = torch.gather(h, 2, idx).contiguous()
            lsp.lsp_view_update(a, k, v, h, acc_t)
            lsp.lsp_view_update(b2, k, v, h_last, acc_t, rows=rows, h_rows=1)
        torch.cuda.synchronize()
        ea, eb = export_state(lsp, a, s), export_state(lsp, b2, s)
        for key in ea:
            assert torch.equal(ea[key], eb[key]), key
        k, v, h = synth.make_features(s, 4, seed=399, device="cuda")
        with pytest.raises(lsp.LspError):
            lsp.lsp_view_update(a, k, v, h, torch.ones(s.C, dtype=torch.int32, device="cuda"), h_rows=2)
    finally:
        lsp.lsp_state_destroy(a)
        lsp.lsp_state_destroy(b2)


def test_incremental_fold_equals_one_shot_fold(lsp):
    """Eq. summary-update is exact: chunking a prefix never changes the result (fp32 tolerance)."""
    s = VU
    cfg = lsp.make_config(s)
    a, b2 = lsp.lsp_state_create(cfg), lsp.lsp_state_create(cfg)
    try:
        G = synth.make_weights(s, seed=4)["G"].cuda()
        lsp.lsp_state_init(a, G)
        lsp.lsp_state_init(b2, G)
        k, v, h = synth.make_features(s, 300, seed=5, device="cuda")
        lsp.lsp_view_update(a, k, v, h, torch.full((s.C,), 300, dtype=torch.int32, device="cuda"))
        for j0 in range(0, 300, 7):
            n = min(7, 300 - j0)
            sl = slice(j0, j0 + n)
            lsp.lsp_view_update(b2, k[:, :, sl].contiguous(), v[:, :, sl].contiguous(),
                                h[:, :, sl].contiguous(), torch.full((s.C,), n, dtype=torch.int32, device="cuda"))
        torch.cuda.synchronize()
        ea, eb = export_state(lsp, a, s), export_state(lsp, b2, s)
        assert torch.equal(ea["t"], eb["t"]) and torch.equal(ea["win_k"], eb["win_k"])
        assert torch.equal(ea["h"], eb["h"])
        torch.testing.assert_close(ea["m"], eb["m"], rtol=0, atol=2e-5)
        torch.testing.assert_close(ea["eta"], eb["eta"], rtol=0, atol=2e-4)
    finally:
        lsp.lsp_state_destroy(a)
        lsp.lsp_state_destroy(b2)


def test_empty_update_is_bit_identical_and_bad_delta_is_reported(lsp):
    s = VU
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        lsp.lsp_state_init(st, synth.make_weights(s, seed=6)["G"].cuda())
        k, v, h = synth.make_features(s, 20, seed=7, device="cuda")
        lsp.lsp_view_update(st, k, v, h, torch.tensor([20, 3, 9], dtype=torch.int32, device="cuda"))
        before = export_state(lsp, st, s)
        lsp.lsp_view_update(st, k, v, h, torch.zeros(s.C, dtype=torch.int32, device="cuda"))
        after = export_state(lsp, st, s)
        for key in before:
            assert torch.equal(before[key], after[key]), key
        # accepted_len beyond the row capacity: reported, request left untouched
        lsp.lsp_view_update(st, k, v, h, torch.tensor([21, 0, 0], dtype=torch.int32, device="cuda"))
        rc, bits = lsp.lsp_get_error(st)
        assert bits & lsp.LSP_DEV_BAD_DELTA and rc == lsp.LSP_ERR_STATE
        again = export_state(lsp, st, s)
        for key in before:
            assert torch.equal(before[key], again[key]), key
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)        # cleared by the previous read
    finally:
        lsp.lsp_state_destroy(st)


SAMP = synth.LspShape("samp", C=5, B=16, L=1, D=1, H=128, nq=1, nkv=1, d=128, F=64, V=32000,
                      W=16, R=16, rc=64)


@pytest.mark.parametrize("temperature", [0.0, 1.0, 0.7])
@pytest.mark.parametrize("dt,C", [("bf16", 5), ("bf16", 16), ("bf16", 20), ("f32", 5)])
def test_sampler_matches_oracle(lsp, temperature, dt, C):
    # bf16 with C <= 16 runs the persistent single-launch kernel, the rest the per-step kernel
    s = SAMP.with_(C=C) if dt == "bf16" else SAMP.with_(dtype="f32", d=64, nq=2, nkv=2)
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        g = torch.Generator().manual_seed(11)
        tdt = s.torch_dtype
        z0 = torch.randn(s.C, s.B, s.V, generator=g) * 2.0
        Ec = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(tdt)
        Wc = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(tdt)
        prev = torch.randint(0, s.V, (s.C,), generator=g, dtype=torch.int32)
        toks = torch.zeros(s.C, s.B, dtype=torch.int32, device="cuda")
        zout = torch.zeros(s.C, s.B, s.V, device="cuda")
        sp = lsp.make_sample_params(temperature, seed=0x1234ABCD5678, rnd=9)
        args = (z0.cuda(), prev.cuda(), Ec.cuda(), Wc.cuda())
        lsp.lsp_sample(st, *args, sp, toks, zout)
        torch.cuda.synchronize()
        toks_g, z_g = toks.cpu().numpy(), f64(zout)
        # a second launch on the same state reproduces the first bit for bit
        toks2 = torch.zeros_like(toks)
        zout2 = torch.zeros_like(zout)
        lsp.lsp_sample(st, *args, sp, toks2, zout2)
        torch.cuda.synchronize()
        assert torch.equal(toks2, toks) and torch.equal(zout2, zout)
        checked = 0
        for b in range(s.C):
            t_o, z_o, marg = oracle.sample_block(f64(z0[b]), int(prev[b]), f64(Ec), f64(Wc), temperature,
                                                 0x1234ABCD5678, 9, b, forced_prev=toks_g[b])
            np.testing.assert_allclose(z_g[b], z_o, rtol=0, atol=2e-5 * np.abs(z_o).max())
            sel = marg > 1e-2
            assert np.array_equal(toks_g[b][sel], t_o[sel]), (b, toks_g[b], t_o, marg)
            checked += sel.sum()
        assert checked >= 0.9 * s.C * s.B
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


def test_sampler_rejects_bad_committed_token(lsp):
    s = SAMP
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        z0 = torch.zeros(s.C, s.B, s.V, device="cuda")
        Ec = torch.zeros(s.V, s.rc, dtype=torch.bfloat16, device="cuda")
        prev = torch.tensor([0, 1, s.V, 3, -5], dtype=torch.int32, device="cuda")
        toks = torch.zeros(s.C, s.B, dtype=torch.int32, device="cuda")
        lsp.lsp_sample(st, z0, prev, Ec, Ec, lsp.make_sample_params(0.0), toks, None)
        rc, bits = lsp.lsp_get_error(st)
        assert bits == lsp.LSP_DEV_BAD_TOKEN and rc == lsp.LSP_ERR_STATE
        assert (toks == 0).all()                     # flat logits: lowest index wins
    finally:
        lsp.lsp_state_destroy(st)
