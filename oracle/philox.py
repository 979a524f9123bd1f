"""Philox4x32-10 counter-based generator (oracle side).

Restated from its published definition: J. K. Salmon, M. A. Moraes, R. O. Dror,
D. E. Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC'11, Sec. 3 (the
Philox S-box with multipliers 0xD2511F53 / 0xCD9E8D57 and Weyl key increments
0x9E3779B9 / 0xBB67AE85, ten rounds).  Vectorised over counters with numpy
uint64 so that 32x32->64-bit products are exact.

The paper under study does not name its sampler RNG; this generator is the
reading chosen for sampled proposals (see the sampler module).
"""
import numpy as np

M0 = np.uint64(0xD2511F53)
M1 = np.uint64(0xCD9E8D57)
W0 = np.uint64(0x9E3779B9)
W1 = np.uint64(0xBB67AE85)
MASK32 = np.uint64(0xFFFFFFFF)
SH32 = np.uint64(32)


def philox4x32_10(ctr, key):
    """ctr: uint array [..., 4]; key: uint array [..., 2] (broadcastable).

    Returns uint32 array [..., 4].
    """
    ctr = np.asarray(ctr, dtype=np.uint64)
    key = np.asarray(key, dtype=np.uint64)
    c0, c1, c2, c3 = (ctr[..., i] & MASK32 for i in range(4))
    k0, k1 = key[..., 0] & MASK32, key[..., 1] & MASK32
    for _ in range(10):
        p0 = M0 * c0
        p1 = M1 * c2
        hi0, lo0 = p0 >> SH32, p0 & MASK32
        hi1, lo1 = p1 >> SH32, p1 & MASK32
        c0, c1, c2, c3 = (hi1 ^ c1 ^ k0) & MASK32, lo1, (hi0 ^ c3 ^ k1) & MASK32, lo0
        k0 = (k0 + W0) & MASK32
        k1 = (k1 + W1) & MASK32
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def sampler_words(seed, rnd, b, i, V):
    """The 32-bit word used for vocabulary entry v at (request b, step i, round rnd).

    Counter = (v >> 2, i, b, rnd), key = (seed low 32 bits, seed high 32 bits),
    output word = v & 3.  Returns uint32 [V].
    """
    v = np.arange(V, dtype=np.uint64)
    nblk = (V + 3) // 4
    blk = np.arange(nblk, dtype=np.uint64)
    ctr = np.stack([blk,
                    np.full(nblk, i, np.uint64),
                    np.full(nblk, b, np.uint64),
                    np.full(nblk, rnd & 0xFFFFFFFF, np.uint64)], axis=-1)
    seed = int(seed)
    key = np.array([seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF], dtype=np.uint64)
    out = philox4x32_10(ctr, key)          # [nblk][4]
    return out[(v >> np.uint64(2)).astype(np.int64), (v & np.uint64(3)).astype(np.int64)]
