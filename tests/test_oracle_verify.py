"""Pins of the oracle's verification rule (Eq. acceptance, Eq. residual).

The anchor is the property the rule exists for: the first emitted token of a
round is distributed exactly as the target's p_1, whatever the proposal q_1,
and a candidate is accepted with probability sum_v min(p_1(v), q_1(v)).  A
swapped p/q, a missing [.]_+ or a wrong acceptance inequality breaks one of
these on a small vocabulary.
"""
import numpy as np
import pytest

from oracle import verify
from oracle.sampler import gumbel

V = 6
ZT = np.array([[1.2, -0.3, 0.5, 2.0, -1.0, 0.0],
               [0.1, 0.2, 0.3, 0.4, 0.5, 0.6]])
ZQ = np.array([[0.2, 1.5, 0.5, 0.3, -0.5, 1.0]])


def _softmax(z):
    e = np.exp(z - z.max())
    return e / e.sum()


def _rounds(zt, zq, T, n, seed0=1000):
    """Draw y_1 ~ q_1 by Gumbel-max (the drafter's rule) and verify; n independent rounds."""
    firsts, accepted = np.zeros(V), 0
    for k in range(n):
        seed = seed0 + k
        y = int(np.argmax(zq[0] / T + gumbel(seed, 7, 0, 0, V)))
        r, tok, _, _ = verify.verify_block(zt, zq, [y], T, seed, 7, 0)
        first = y if r >= 1 else tok
        firsts[first] += 1
        accepted += r
    return firsts / n, accepted / n


@pytest.mark.parametrize("T", [1.0, 0.6])
def test_first_emitted_token_follows_the_target(T):
    n = 6000
    freq, acc = _rounds(ZT, ZQ, T, n)
    p1 = _softmax(ZT[0] / T)
    q1 = _softmax(ZQ[0] / T)
    # 5 standard errors of a multinomial frequency
    assert np.all(np.abs(freq - p1) <= 5 * np.sqrt(p1 * (1 - p1) / n) + 1e-3), (freq, p1)
    # the proposal alone would be far off: the test can tell p from q
    assert np.max(np.abs(q1 - p1)) > 0.1
    a = np.minimum(p1, q1).sum()
    assert abs(acc - a) <= 5 * np.sqrt(a * (1 - a) / n), (acc, a)


def test_identical_distributions_accept_every_candidate_and_draw_the_bonus_from_p():
    zt = np.array([[0.3, 0.1, -0.2, 0.9, 0.0, 0.4],
                   [0.3, 0.1, -0.2, 0.9, 0.0, 0.4],
                   [1.0, -1.0, 0.5, 0.2, 0.0, -0.5]])
    zq = zt[:2].copy()
    n = 4000
    bonus = np.zeros(V)
    for k in range(n):
        y = [int(np.argmax(zq[i] + gumbel(50 + k, 3, 1, i, V))) for i in range(2)]
        r, tok, _, _ = verify.verify_block(zt, zq, y, 1.0, 50 + k, 3, 1)
        assert r == 2                                   # alpha = 1 whenever p = q
        bonus[tok] += 1
    p3 = _softmax(zt[2])
    assert np.all(np.abs(bonus / n - p3) <= 5 * np.sqrt(p3 * (1 - p3) / n) + 1e-3)


def test_a_candidate_the_target_forbids_is_always_rejected_and_never_redrawn():
    zt = np.array([[0.0, -np.inf, 0.5, 0.2, 0.1, 0.0],
                   [0.0, 0.0, 0.0, 0.0, 0.0, 0.0]])
    zq = np.array([[0.0, 3.0, 0.0, 0.0, 0.0, 0.0]])
    for k in range(200):
        r, tok, _, _ = verify.verify_block(zt, zq, [1], 1.0, 10 + k, 0, 0)
        assert r == 0 and tok != 1


def test_greedy_accepts_the_matching_prefix_and_emits_the_target_argmax():
    zt = np.array([[0.0, 1.0, 0.0, 0.0, 0.0, 0.0],
                   [0.0, 0.0, 2.0, 0.0, 0.0, 0.0],
                   [0.0, 0.0, 0.0, 3.0, 3.0, 0.0],      # tie: lowest index
                   [5.0, 0.0, 0.0, 0.0, 0.0, 0.0]])
    zq = np.zeros((3, V))
    assert verify.verify_block(zt, zq, [1, 2, 3], 0.0, 0, 0, 0)[:2] == (3, 0)
    assert verify.verify_block(zt, zq, [1, 2, 4], 0.0, 0, 0, 0)[:2] == (2, 3)
    assert verify.verify_block(zt, zq, [1, 5, 3], 0.0, 0, 0, 0)[:2] == (1, 2)
    assert verify.verify_block(zt, zq, [0, 2, 3], 0.0, 0, 0, 0)[:2] == (0, 1)


def test_verification_randomness_is_a_separate_philox_stream():
    # acceptance and draw counters differ from every drafting counter (second word < 2^30)
    from oracle.philox import sampler_words
    d = sampler_words(5, 1, 0, 0, 8)
    a = sampler_words(5, 1, 0, verify.ACCEPT_STREAM, 8)
    g = sampler_words(5, 1, 0, verify.DRAW_STREAM, 8)
    assert not np.array_equal(d, a) and not np.array_equal(d, g) and not np.array_equal(a, g)
    u = verify.accept_uniform(5, 1, 0, 0)
    assert 0.0 < u < 1.0 and u == (float(a[0] >> np.uint32(9)) + 0.5) * 2.0 ** -23


def test_accepted_length_is_truncated_geometric_in_alpha():
    """With the same (p, q) at every position, each candidate is accepted with probability
    alpha = sum_v min(p(v), q(v)) independently of the others, and the round stops at the
    first rejection: P(r = k) = alpha^k (1 - alpha) for k < B and P(r = B) = alpha^B.
    Accepting past a rejection, or a per-position ratio other than p/q, breaks it."""
    B, n, T = 3, 6000, 1.0
    zq1 = ZQ[0]
    zt = np.stack([ZT[0]] * (B + 1))
    zq = np.stack([zq1] * B)
    hist = np.zeros(B + 1)
    for k in range(n):
        seed = 7000 + k
        y = [int(np.argmax(zq[i] / T + gumbel(seed, 5, 2, i, V))) for i in range(B)]
        r, _, _, _ = verify.verify_block(zt, zq, y, T, seed, 5, 2)
        hist[r] += 1
    a = np.minimum(_softmax(ZT[0] / T), _softmax(zq1 / T)).sum()
    want = np.array([a ** j * (1 - a) for j in range(B)] + [a ** B])
    got = hist / n
    assert np.all(np.abs(got - want) <= 5 * np.sqrt(want * (1 - want) / n) + 1e-3), (got, want)
    assert 0.2 < a < 0.8                     # every length has weight: the law is visible
