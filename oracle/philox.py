"""Philox4x32-10 counter-based generator (Salmon, Moraes, Dror, Shaw,
"Parallel random numbers: as easy as 1, 2, 3", SC 2011) -- TEST
INFRASTRUCTURE ONLY, written from the published definition: ten rounds of
two 32x32->64-bit multiplies by M0 = 0xD2511F53 and M1 = 0xCD9E8D57, with the
key bumped by the Weyl constants W0 = 0x9E3779B9, W1 = 0xBB67AE85 between
rounds.  Vectorised over counters with NumPy uint64 arithmetic.

Used by the oracle for temperature sampling: the same generator, implemented
independently on the device, gives the Gumbel noise of both sides.
"""
from __future__ import annotations

import numpy as np

M0, M1 = 0xD2511F53, 0xCD9E8D57
W0, W1 = 0x9E3779B9, 0xBB67AE85
MASK = 0xFFFFFFFF


def philox4x32_10(c0, c1, c2, c3, k0: int, k1: int):
    """Four uint32 outputs for each counter (c0, c1, c2, c3) under key (k0, k1)."""
    c = [np.asarray(x, dtype=np.uint64) & MASK for x in (c0, c1, c2, c3)]
    k0, k1 = np.uint64(k0 & MASK), np.uint64(k1 & MASK)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + np.uint64(W0)) & np.uint64(MASK)
            k1 = (k1 + np.uint64(W1)) & np.uint64(MASK)
        p0 = np.uint64(M0) * c[0]
        p1 = np.uint64(M1) * c[2]
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK)
        c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return [x.astype(np.uint32) for x in c]


def uniform23(r) -> np.ndarray:
    """(floor(r / 2^9) + 0.5) / 2^23: a uniform value in the open interval (0, 1),
    an odd multiple of 2^-24, which float32 and float64 both represent exactly
    (the largest is 1 - 2^-24, so float32 never rounds it to 1)."""
    return ((np.asarray(r, dtype=np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) / 8388608.0


def gumbel_noise(seed: int, rows: int, vocab: int) -> np.ndarray:
    """g[m, v] = -log(-log(u)) with u from counter (v, m // 4, 0, 0), output m % 4,
    key (seed mod 2^32, seed // 2^32).  Shape [rows, vocab], float64."""
    v = np.arange(vocab, dtype=np.uint64)
    g = np.empty((rows, vocab), dtype=np.float64)
    k0, k1 = seed & MASK, (seed >> 32) & MASK
    for q in range((rows + 3) // 4):
        outs = philox4x32_10(v, np.full(vocab, q, dtype=np.uint64), 0, 0, k0, k1)
        for j in range(4):
            m = 4 * q + j
            if m < rows:
                g[m] = -np.log(-np.log(uniform23(outs[j])))
    return g
