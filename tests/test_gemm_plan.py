"""The projection GEMM's launch plan, host logic only (no GPU): the split-K
factor and token groups the drafter takes at the Qwen3-8B round on a 152-SM
GB300, and the token-group invariants the kernel relies on (every token row
in exactly one group, no empty group)."""
import pytest

GU = dict(N=12288, K=4096, swiglu=1)


@pytest.fixture(scope="module")
def lsp():
    from paper_2609_37029_gb300 import build
    build.build()
    from paper_2609_37029_gb300 import lsp as mod
    return mod


def plan(lsp, M, N, K, swiglu=0, sms=152, dtype=None):
    return lsp.lsp_gemm_plan_info(lsp.LSP_DTYPE_BF16 if dtype is None else dtype, M, N, K, swiglu, sms)


def test_qwen3_8b_round_plan(lsp):
    # M = C x B = 256 block tokens; the boundary fusion runs on the C = 16 requests
    assert plan(lsp, 16, 4096, 5 * 4096) == (9, 1, 16)      # boundary fusion (5 tapped layers)
    assert plan(lsp, 256, 6144, 4096) == (3, 1, 256)        # q/k/v (32 + 2 x 8 heads of 128)
    assert plan(lsp, 256, 4096, 4096) == (4, 1, 256)        # o_proj
    assert plan(lsp, 256, 4096, 12288) == (9, 1, 256)       # down
    assert plan(lsp, 256, **GU) == (1, 2, 128)              # gate/up: two token groups


@pytest.mark.parametrize("sms,groups", [(152, 2), (96, 2), (95, 1), (192, 2), (193, 1)])
def test_gate_up_groups_only_for_an_underfilled_single_wave(lsp, sms, groups):
    """192 gate/up tiles: two groups when num_sms <= 192 <= 2 num_sms (at least a wave of one
    CTA per SM, less than a wave of two)."""
    assert plan(lsp, 256, sms=sms, **GU)[1] == groups
    assert plan(lsp, 112, sms=sms, **GU)[1] == 1             # B = 7 (M = 112): one group


@pytest.mark.parametrize("N", [12288, 9728, 19456])
def test_token_groups_cover_every_row_once(lsp, N):
    """Over every token count, the plan's groups cover each row once with no empty
    group; the other projections take two groups exactly when M > 256 (one 256-token
    tile per CTA instead of a 512-column accumulator)."""
    for M in range(1, 513):
        for sw in (1, 0):
            _, g, rows = plan(lsp, M, N, 1024, swiglu=sw)
            assert 1 <= g <= 2 and rows % 16 == 0 and rows <= 512
            assert g * rows >= M > (g - 1) * rows, (M, g, rows)   # covered, last group not empty
            assert g == 1 or M >= 16 * g
            assert rows <= 256 or M <= 256
        assert plan(lsp, M, N, 1024)[1] == (2 if M > 256 else 1)


def test_bad_arguments(lsp):
    for args in [(0, 128, 128, 0, 152), (513, 128, 128, 0, 152), (16, 0, 128, 0, 152),
                 (16, 128, 0, 0, 152), (16, 128, 128, 0, 0)]:
        with pytest.raises(lsp.LspError):
            lsp.lsp_gemm_plan_info(lsp.LSP_DTYPE_BF16, *args)
    with pytest.raises(lsp.LspError):
        lsp.lsp_gemm_plan_info(7, 16, 128, 128, 0, 152)
