"""lsp_sample_noalloc: the sampler for callers that cannot allocate device memory.

Such a caller (one running under another framework's caching allocator that
has reserved the device, or one that must not create an lsp_state) passes only
its inputs and outputs; the scratch lives in a fixed array inside the library.
This checks, through the C ABI, that two calls in a row give the same tokens
and corrected logits as lsp_sample, the existing entry point, on the same
inputs -- on each kernel the call can take: the one-launch bf16 loop (C <= 16,
r_c = 64), the per-step kernels (C > 16, or another rank), and the fp32 loop --
and that a shape at the scratch limit is accepted and one row past it refused.
The file is named so that pytest collects it last.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2609_37029_gb300 import synth
from tests.gpu_common import lsp_lib

pytestmark = pytest.mark.gpu


def _shape(C, B, V, rc, dtype):
    # only C, B, V, rc and the storage type matter to the sampler; the rest is any valid config
    heads = dict(nq=1, nkv=1, d=128) if dtype == "bf16" else dict(nq=2, nkv=2, d=64)
    return synth.LspShape("noalloc", C=C, B=B, L=1, D=1, H=128, F=64, V=V, W=16, R=16, rc=rc,
                          dtype=dtype, **heads)


def _inputs(s, seed):
    g = torch.Generator().manual_seed(seed)
    z0 = (torch.randn(s.C, s.B, s.V, generator=g) * 2.0).cuda()
    Ec = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(s.torch_dtype).cuda()
    Wc = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(s.torch_dtype).cuda()
    prev = torch.randint(0, s.V, (s.C,), generator=g, dtype=torch.int32).cuda()
    return z0, Ec, Wc, prev


CASES = {
    "bf16-one-launch": (16, 16, 32000, 64, "bf16"),
    "bf16-per-step-C20": (20, 16, 32000, 64, "bf16"),
    "bf16-per-step-rc48": (8, 16, 4096, 48, "bf16"),
    "f32-one-launch": (4, 16, 8192, 32, "f32"),
}


@pytest.mark.parametrize("case", list(CASES))
def test_noalloc_sampler_matches_lsp_sample_on_two_calls_in_a_row(case):
    lsp = lsp_lib()
    s = _shape(*CASES[case])
    code = lsp.LSP_DTYPE_BF16 if s.dtype == "bf16" else lsp.LSP_DTYPE_F32
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        for call, (temperature, seed) in enumerate([(1.0, 21), (0.0, 22)]):
            z0, Ec, Wc, prev = _inputs(s, seed)
            sp = lsp.make_sample_params(temperature, seed=0xC0FFEE + call, rnd=call)
            ref_t = torch.zeros(s.C, s.B, dtype=torch.int32, device="cuda")
            ref_z = torch.zeros(s.C, s.B, s.V, device="cuda")
            lsp.lsp_sample(st, z0, prev, Ec, Wc, sp, ref_t, ref_z)
            got_t = torch.full((s.C, s.B), -7, dtype=torch.int32, device="cuda")
            got_z = torch.zeros(s.C, s.B, s.V, device="cuda")
            err = torch.zeros(1, dtype=torch.int32, device="cuda")
            lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, code, s.C, s.B, s.V, s.rc, sp, got_t, got_z, err)
            torch.cuda.synchronize()
            assert torch.equal(got_t, ref_t), (case, call)
            torch.testing.assert_close(got_z, ref_z, rtol=0, atol=2e-5 * ref_z.abs().max().item())
            assert int(err.item()) == 0
        assert lsp.lsp_get_error(st) == (lsp.LSP_OK, 0)
    finally:
        lsp.lsp_state_destroy(st)


def _limit_rows(C, num_sms):
    """Largest B whose scratch fits the 512 KiB array (the formula lsp.h states)."""
    a256 = lambda x: (x + 255) // 256 * 256
    nblk = min(2 * num_sms, 512)
    B = 0
    while a256(16 * nblk * C) + a256(2052 * (B + 1)) <= 512 * 1024:
        B += 1
    return B


def test_noalloc_sampler_at_the_scratch_limit():
    """C = 64 at the largest B the array holds: accepted, greedy tokens equal the oracle's
    wherever its top-1/top-2 margin exceeds 1e-2 (teacher-forced), no device error; one
    more row is refused with LSP_ERR_SHAPE before anything is enqueued."""
    lsp = lsp_lib()
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    B = _limit_rows(64, sms)
    assert B >= 1
    s = _shape(64, B, 1024, 64, "bf16")
    z0, Ec, Wc, prev = _inputs(s, 31)
    sp = lsp.make_sample_params(0.0)
    toks = torch.full((s.C, s.B), -7, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, lsp.LSP_DTYPE_BF16, s.C, s.B, s.V, s.rc, sp, toks, None, err)
    torch.cuda.synchronize()
    assert int(err.item()) == 0
    t_g = toks.cpu().numpy()
    Ec64, Wc64 = Ec.double().cpu().numpy(), Wc.double().cpu().numpy()
    z64, p64 = z0.double().cpu().numpy(), prev.cpu().numpy()
    for b in (0, 37, 63):
        t_o, _, marg = oracle.sample_block(z64[b], int(p64[b]), Ec64, Wc64, 0.0, 0, 0, b, forced_prev=t_g[b])
        sel = marg > 1e-2
        assert sel.sum() >= 0.5 * s.B
        assert np.array_equal(t_g[b][sel], t_o[sel]), b
    with pytest.raises(lsp.LspError) as e:
        lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, lsp.LSP_DTYPE_BF16, s.C, B + 1, s.V, s.rc, sp, toks)
    assert e.value.status == lsp.LSP_ERR_SHAPE


def test_noalloc_sampler_rejects_oversized_and_bad_arguments():
    lsp = lsp_lib()
    s = _shape(16, 16, 32000, 64, "bf16")
    z0, Ec, Wc, prev = _inputs(s, 23)
    toks = torch.zeros(s.C, s.B, dtype=torch.int32, device="cuda")
    sp = lsp.make_sample_params(1.0)
    with pytest.raises(lsp.LspError) as e:
        lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, lsp.LSP_DTYPE_BF16, 65, s.B, s.V, s.rc, sp, toks)
    assert e.value.status == lsp.LSP_ERR_SHAPE
    with pytest.raises(lsp.LspError) as e:
        lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, 7, s.C, s.B, s.V, s.rc, sp, toks)
    assert e.value.status == lsp.LSP_ERR_ARG
