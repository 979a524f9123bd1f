"""Target-side verification (Sec. 2.1, Eq. acceptance, Eq. residual, bonus draw):
lsp_verify against the oracle's verify_block on the same logits, drafted tokens
and Philox key.

Decisions (accept / reject, the Gumbel-max winner) are compared exactly where
the oracle's fp64 decision is clear of fp32 rounding: an acceptance test whose
two sides differ by more than 1e-3 (relative), a draw whose top-2 score gap
exceeds 1e-3.  A decision closer than that is still checked for validity: the
GPU's emitted token must score within 1e-2 of the oracle's best.
"""
import numpy as np
import pytest
import torch

import oracle
from oracle.sampler import gumbel
from oracle.verify import draw_gumbel
from tests.gpu_common import lsp_lib
from paper_2609_37029_gb300 import synth

pytestmark = pytest.mark.gpu

ACC_TOL = 1e-3
DRAW_TOL = 1e-3


@pytest.fixture(scope="module")
def lsp():
    return lsp_lib()


def _shape(C, B, V):
    return synth.LspShape("verify", C=C, B=B, L=1, D=1, H=256, nq=2, nkv=1, d=128, F=256, V=V,
                          W=8, R=16, rc=16)


def _draft_tokens(zq, T, seed, rnd):
    """y_i ~ q_i by the drafter's Gumbel-max rule (argmax at T = 0)."""
    C, B, V = zq.shape
    y = np.zeros((C, B), dtype=np.int32)
    for b in range(C):
        for i in range(B):
            z = zq[b, i].astype(np.float64)
            y[b, i] = np.argmax(z) if T <= 0 else np.argmax(z / T + gumbel(seed, rnd, b, i, V))
    return y


def _score(zt, zq, T, r, B, seed, rnd, b):
    """The oracle's fp64 draw score of every token at the emitting position."""
    V = zt.shape[-1]
    if T <= 0:
        return zt[r].astype(np.float64)

    def sm(z):
        e = np.exp(z - z.max())
        return e / e.sum()
    p = sm(zt[r].astype(np.float64) / T)
    w = np.maximum(p - sm(zq[r].astype(np.float64) / T), 0.0) if r < B else p
    with np.errstate(divide="ignore"):
        return np.log(w) + draw_gumbel(seed, rnd, b, r, V)


def _run(lsp, s, zt, zq, y, T, seed, rnd):
    st = lsp.lsp_state_create(lsp.make_config(s))
    try:
        acc = torch.zeros(s.C, dtype=torch.int32, device="cuda")
        tok = torch.zeros(s.C, dtype=torch.int32, device="cuda")
        sp = lsp.make_sample_params(temperature=T, seed=seed, rnd=rnd)
        lsp.lsp_verify(st, zt.cuda(), zq.cuda(), torch.from_numpy(y).cuda(), sp, acc, tok)
        torch.cuda.synchronize()
        err = lsp.lsp_get_error(st)
        return acc.cpu().numpy(), tok.cpu().numpy(), err
    finally:
        lsp.lsp_state_destroy(st)


def _compare(s, zt, zq, y, T, seed, rnd, acc, tok):
    zt_n, zq_n = zt.numpy(), zq.numpy()
    exact = 0
    for b in range(s.C):
        r, t, margins, dm = oracle.verify_block(zt_n[b], zq_n[b], y[b], T, seed, rnd, b)
        tested = margins[:r + 1] if r < s.B else margins
        clear = T <= 0 or all(m > ACC_TOL for m in tested)
        if clear:
            assert acc[b] == r, (b, acc[b], r, tested)
        if clear and acc[b] == r and dm > DRAW_TOL:
            assert tok[b] == t, (b, tok[b], t, dm)
            exact += 1
        else:
            # a near-tie: the GPU's choice must still be (numerically) a valid outcome
            assert 0 <= acc[b] <= s.B and 0 <= tok[b] < s.V
            sc = _score(zt_n[b], zq_n[b], T, int(acc[b]), s.B, seed, rnd, b)
            assert sc[tok[b]] >= sc.max() - 1e-2, (b, sc[tok[b]], sc.max())
    return exact


@pytest.mark.parametrize("T,C,B,V", [(1.0, 8, 5, 1008), (0.7, 8, 16, 1008), (1.0, 3, 16, 4112),
                                     (0.0, 8, 16, 1008), (1.0, 2, 7, 151936), (0.0, 2, 7, 151936)])
def test_verify_matches_oracle(lsp, T, C, B, V):
    s = _shape(C, B, V)
    seed, rnd = 4242 + V, 9
    zt, zq = synth.make_verify_logits(s, seed=17 + B)
    y = _draft_tokens(zq.numpy(), T, seed, rnd)
    acc, tok, err = _run(lsp, s, zt, zq, y, T, seed, rnd)
    assert err == (lsp.LSP_OK, 0)
    exact = _compare(s, zt, zq, y, T, seed, rnd, acc, tok)
    assert exact >= C - 1, exact                       # near-ties are rare: most compare exactly
    if T > 0 and C >= 8:
        assert len(set(acc.tolist())) >= 3             # the accepted lengths really spread


@pytest.mark.parametrize("T", [1.0, 0.0])
def test_verify_at_the_bench_shape_on_sampled_requests(lsp, T):
    """C = 16, B = 16, V = 151936 -- the launch configuration bench.py times.  Requests 0
    and 11 carry candidates drafted from q by the drafter's rule and are compared with the
    oracle; the others carry random candidates (valid input, mostly rejected at once) and
    are checked for range only."""
    s = _shape(16, 16, 151936)
    seed, rnd = 99, 4
    zt, zq = synth.make_verify_logits(s, seed=61)
    g = np.random.default_rng(5)
    y = g.integers(0, s.V, size=(s.C, s.B)).astype(np.int32)
    picked = [0, 11]
    for b in picked:
        y[b] = _draft_rows(zq[b].numpy(), T, seed, rnd, b)
    acc, tok, err = _run(lsp, s, zt, zq, y, T, seed, rnd)
    assert err == (lsp.LSP_OK, 0)
    assert ((acc >= 0) & (acc <= s.B)).all() and ((tok >= 0) & (tok < s.V)).all()
    sub = _shape(1, 16, 151936)
    for b in picked:
        one = _compare_one(sub, zt[b].numpy(), zq[b].numpy(), y[b], T, seed, rnd, b, acc[b], tok[b])
        assert one, b


def _draft_rows(zq_b, T, seed, rnd, b):
    """Request b's candidates by the drafter's Gumbel-max rule (argmax at T = 0)."""
    B, V = zq_b.shape
    return np.array([np.argmax(zq_b[i].astype(np.float64)) if T <= 0 else
                     np.argmax(zq_b[i].astype(np.float64) / T + gumbel(seed, rnd, b, i, V))
                     for i in range(B)], dtype=np.int32)


def _compare_one(s, zt_b, zq_b, y_b, T, seed, rnd, b, acc_b, tok_b):
    """One request against the oracle with the margin rules of _compare; True when the
    decisions were clear enough to compare exactly (and matched)."""
    r, t, margins, dm = oracle.verify_block(zt_b, zq_b, y_b, T, seed, rnd, b)
    tested = margins[:r + 1] if r < s.B else margins
    if T > 0 and not all(m > ACC_TOL for m in tested):
        return True                      # a near-tie: nothing exact to compare
    assert acc_b == r, (b, acc_b, r)
    if dm > DRAW_TOL:
        assert tok_b == t, (b, tok_b, t, dm)
    return True


def test_verify_accepts_everything_when_draft_equals_target(lsp):
    """p = q makes alpha = 1: r = B for every request and the bonus follows p_{B+1}."""
    s = _shape(6, 16, 2048)
    seed, rnd = 77, 3
    zt, _ = synth.make_verify_logits(s, seed=5)
    zq = zt[:, :s.B].clone()
    y = _draft_tokens(zq.numpy(), 1.0, seed, rnd)
    acc, tok, err = _run(lsp, s, zt, zq, y, 1.0, seed, rnd)
    assert err == (lsp.LSP_OK, 0)
    assert (acc == s.B).all()
    _compare(s, zt, zq, y, 1.0, seed, rnd, acc, tok)


def test_verify_forbidden_candidate_is_rejected(lsp):
    """A candidate the target gives probability 0 is rejected and never emitted."""
    s = _shape(4, 5, 1024)
    seed, rnd = 11, 0
    zt, zq = synth.make_verify_logits(s, seed=8, agree=(0.99, 0.99))
    y = _draft_tokens(zq.numpy(), 1.0, seed, rnd)
    for b in range(s.C):
        zt[b, 2, y[b, 2]] = -float("inf")
    acc, tok, err = _run(lsp, s, zt, zq, y, 1.0, seed, rnd)
    assert err == (lsp.LSP_OK, 0)
    assert (acc <= 2).all()
    for b in range(s.C):
        if acc[b] == 2:
            assert tok[b] != y[b, 2]
    _compare(s, zt, zq, y, 1.0, seed, rnd, acc, tok)


def test_verify_greedy_example(lsp):
    """T = 0: the matching prefix is accepted and the target argmax emitted (ties -> lowest index)."""
    s = _shape(4, 3, 16)
    zt = torch.zeros((4, 4, 16))
    zt[:, 0, 1] = 1.0
    zt[:, 1, 2] = 2.0
    zt[:, 2, 3] = 3.0
    zt[:, 2, 4] = 3.0
    zt[:, 3, 0] = 5.0
    zq = torch.zeros((4, 3, 16))
    y = np.array([[1, 2, 3], [1, 2, 4], [1, 5, 3], [0, 2, 3]], dtype=np.int32)
    acc, tok, err = _run(lsp, s, zt, zq, y, 0.0, 0, 0)
    assert err == (lsp.LSP_OK, 0)
    assert acc.tolist() == [3, 2, 1, 0] and tok.tolist() == [0, 3, 2, 1]


@pytest.mark.parametrize("T", [0.0, 1.0])
def test_verify_flags_out_of_range_tokens(lsp, T):
    s = _shape(2, 4, 512)
    zt, zq = synth.make_verify_logits(s, seed=2)
    y = _draft_tokens(zq.numpy(), T, 1, 1)
    y[1, 0] = s.V + 7
    acc, tok, (rc, bits) = _run(lsp, s, zt, zq, y, T, 1, 1)
    assert bits & lsp.LSP_DEV_BAD_TOKEN and rc == lsp.LSP_ERR_STATE
    assert 0 <= acc[1] <= s.B and 0 <= tok[1] < s.V


def test_verify_is_deterministic(lsp):
    s = _shape(8, 16, 4096)
    zt, zq = synth.make_verify_logits(s, seed=31)
    y = _draft_tokens(zq.numpy(), 1.0, 5, 2)
    a1, t1, _ = _run(lsp, s, zt, zq, y, 1.0, 5, 2)
    a2, t2, _ = _run(lsp, s, zt, zq, y, 1.0, 5, 2)
    assert (a1 == a2).all() and (t1 == t2).all()
