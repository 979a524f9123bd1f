"""Pins for the oracle's correction and sampler (Eq. markov, Eq. proposal-factorization) -- CPU only."""
import os

import numpy as np
import pytest
from scipy import stats
from scipy.special import softmax

from oracle import philox, sampler

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _kat():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append([int(x, 16) for x in line.split()])
    return np.array(rows, dtype=np.uint64)


def test_philox_known_answer_vectors():
    kat = _kat()
    out = philox.philox4x32_10(kat[:, 0:4], kat[:, 4:6])
    np.testing.assert_array_equal(out.astype(np.uint64), kat[:, 6:10])


def test_sampler_words_layout():
    """Word for v is lane v & 3 of the block with counter (v >> 2, i, b, round)."""
    w = philox.sampler_words(0x1234567890ABCDEF, 5, 3, 2, 10)
    blk = philox.philox4x32_10(np.array([[2, 2, 3, 5]]), np.array([[0x90ABCDEF, 0x12345678]]))[0]
    assert list(w[8:10]) == list(blk[0:2])


def test_gumbel_noise_is_finite_and_standard():
    g = np.concatenate([sampler.gumbel(7, r, 0, 0, 4096) for r in range(8)])
    assert np.isfinite(g).all()
    # Gumbel(0, 1): mean = Euler-Mascheroni, variance = pi^2 / 6
    assert abs(g.mean() - np.euler_gamma) < 0.03
    assert abs(g.var() - np.pi ** 2 / 6) < 0.06
    ks = stats.kstest(g, stats.gumbel_r.cdf)
    assert ks.pvalue > 1e-3


def test_greedy_without_correction_is_rowwise_argmax():
    rng = np.random.default_rng(1)
    B, V, rc = 6, 50, 4
    z0 = rng.standard_normal((B, V))
    toks, zs, _ = sampler.sample_block(z0, 3, rng.standard_normal((V, rc)), np.zeros((V, rc)),
                                       0.0, 7, 0, 0)
    np.testing.assert_array_equal(toks, z0.argmax(axis=1))
    np.testing.assert_array_equal(zs, z0)


def test_markov_correction_conditions_on_the_previous_token():
    """E_c(y) one-hot and W_c a shift: the correction pushes token y+1 after y.

    With flat base logits the greedy chain must read a+1, a+2, ... (y_0 = a).
    """
    V = 12
    Ec = np.eye(V)
    Wc = np.roll(np.eye(V), 1, axis=0) * 5.0     # (W_c E_c(y))[v] = 5 [v == y+1]
    z0 = np.zeros((7, V))
    toks, zs, _ = sampler.sample_block(z0, 9, Ec, Wc, 0.0, 1, 0, 0)
    np.testing.assert_array_equal(toks, [(9 + i + 1) % V for i in range(7)])
    assert zs[0, 10] == 5.0 and zs[0].sum() == 5.0
    # teacher forcing: step i conditions on forced_prev[i-1]
    forced = np.array([0, 4, 4, 4, 4, 4, 4])
    toks_f, _, _ = sampler.sample_block(z0, 9, Ec, Wc, 0.0, 1, 0, 0, forced_prev=forced)
    np.testing.assert_array_equal(toks_f, [10, 1, 5, 5, 5, 5, 5])


def test_ties_go_to_lowest_index():
    z0 = np.zeros((2, 9))
    z0[:, 3] = z0[:, 6] = 1.0
    toks, _, margins = sampler.sample_block(z0, 0, np.zeros((9, 2)), np.zeros((9, 2)), 0.0, 1, 0, 0)
    assert list(toks) == [3, 3] and margins[0] == 0.0


@pytest.mark.parametrize("temperature", [1.0, 0.5])
def test_gumbel_max_frequencies_follow_softmax(temperature):
    """chi^2: y ~ softmax(z / T) over 2e4 independent counters (Eq. proposal-factorization)."""
    V, n = 16, 20000
    rng = np.random.default_rng(3)
    z = rng.standard_normal(V) * 1.5
    counts = np.zeros(V)
    zero = np.zeros((V, 1))
    for r in range(n // 8):
        toks, _, _ = sampler.sample_block(np.tile(z, (8, 1)), 0, zero, zero, temperature, 11, r, 5)
        np.add.at(counts, toks, 1)
    expected = softmax(z / temperature) * n
    chi2 = ((counts - expected) ** 2 / expected).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-4
