"""lsp_sample_noalloc: the sampler for callers that cannot allocate device memory.

Such a caller (one running under another framework's caching allocator that
has reserved the device, or one that must not create an lsp_state) passes only
its inputs and outputs; the scratch lives in a fixed array inside the library.
This checks, through the C ABI, that two calls in a row give the same tokens
and corrected logits as lsp_sample, the existing entry point, on the same
inputs.  The file is named so that pytest collects it last.
"""
import pytest
import torch

from paper_2609_37029_gb300 import synth
from tests.gpu_common import lsp_lib

pytestmark = pytest.mark.gpu

SHAPE = synth.LspShape("noalloc", C=16, B=16, L=1, D=1, H=128, nq=1, nkv=1, d=128, F=64,
                       V=32000, W=16, R=16, rc=64)


def _inputs(s, seed):
    g = torch.Generator().manual_seed(seed)
    z0 = (torch.randn(s.C, s.B, s.V, generator=g) * 2.0).cuda()
    Ec = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(torch.bfloat16).cuda()
    Wc = (torch.randn(s.V, s.rc, generator=g) * 0.5).to(torch.bfloat16).cuda()
    prev = torch.randint(0, s.V, (s.C,), generator=g, dtype=torch.int32).cuda()
    return z0, Ec, Wc, prev


def test_noalloc_sampler_matches_lsp_sample_on_two_calls_in_a_row():
    lsp = lsp_lib()
    s = SHAPE
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
            lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, lsp.LSP_DTYPE_BF16, s.C, s.B, s.V, s.rc, sp,
                                   got_t, got_z, err)
            torch.cuda.synchronize()
            assert torch.equal(got_t, ref_t), call
            torch.testing.assert_close(got_z, ref_z, rtol=0, atol=2e-5 * ref_z.abs().max().item())
            assert int(err.item()) == 0
    finally:
        lsp.lsp_state_destroy(st)


def test_noalloc_sampler_rejects_oversized_and_bad_arguments():
    lsp = lsp_lib()
    s = SHAPE
    z0, Ec, Wc, prev = _inputs(s, 23)
    toks = torch.zeros(s.C, s.B, dtype=torch.int32, device="cuda")
    sp = lsp.make_sample_params(1.0)
    with pytest.raises(lsp.LspError) as e:
        lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, lsp.LSP_DTYPE_BF16, 65, s.B, s.V, s.rc, sp, toks)
    assert e.value.status == lsp.LSP_ERR_SHAPE
    with pytest.raises(lsp.LspError) as e:
        lsp.lsp_sample_noalloc(z0, prev, Ec, Wc, 7, s.C, s.B, s.V, s.rc, sp, toks)
    assert e.value.status == lsp.LSP_ERR_ARG
