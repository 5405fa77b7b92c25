"""Philox4x32-10 counter-based generator (test infrastructure).

Written from the published definition (Salmon, Moraes, Dror, Shaw, "Parallel
random numbers: as easy as 1, 2, 3", SC 2011): a 4 x 32-bit counter is
scrambled by ten rounds of two 32 x 32 -> 64-bit multiplies, the key being
advanced by two Weyl constants between rounds.  Vectorised over arrays of
counters with uint64 arithmetic for the multiplies.
"""
from __future__ import annotations

import numpy as np

M0, M1 = np.uint64(0xD2511F53), np.uint64(0xCD9E8D57)   # round multipliers
W0, W1 = np.uint64(0x9E3779B9), np.uint64(0xBB67AE85)   # key increments (Weyl sequence)
MASK = np.uint64(0xFFFFFFFF)


def philox4x32_10(c0, c1, c2, c3, k0, k1):
    """Ten Philox rounds; all arguments broadcastable integer arrays (< 2^32).
    Returns the four 32-bit output words as uint64 arrays."""
    c0, c1, c2, c3 = (np.asarray(x, dtype=np.uint64) & MASK for x in (c0, c1, c2, c3))
    k0 = np.asarray(k0, dtype=np.uint64) & MASK
    k1 = np.asarray(k1, dtype=np.uint64) & MASK
    for rnd in range(10):
        if rnd:
            k0 = (k0 + W0) & MASK
            k1 = (k1 + W1) & MASK
        p0 = M0 * c0                      # < 2^64: exact in uint64
        p1 = M1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & MASK
        hi1, lo1 = p1 >> np.uint64(32), p1 & MASK
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def uniform_open(word):
    """A 32-bit word -> the float in (0, 1) ((word >> 9) + 1/2) / 2^23 (exact in fp32 and fp64)."""
    return ((np.asarray(word, dtype=np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) / 8388608.0
