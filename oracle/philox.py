"""Philox4x32-10 counter-based RNG, oracle side (test infrastructure only).

Written from the published definition: J. K. Salmon, M. A. Moraes, R. O. Dror,
D. E. Shaw, "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11, Sec. 3.
A Philox-4x32 round multiplies counter words 0 and 2 by two fixed odd
constants, keeps both 32-bit halves of each 64-bit product and mixes the high
halves with the other two counter words and the round key; the round key is
bumped by two Weyl constants between rounds.  Ten rounds are applied.

The sampler's uniform draw is defined here (the paper is silent on its RNG):
key = (seed low 32 bits, seed high 32 bits), counter = (step low 32 bits,
step high 32 bits, 0, 0); u = (output word 0 >> 8) * 2**-24, which lies in
[0, 1) and is exactly representable in fp32 and fp64.

Pinned by the published known-answer vectors (tests/golden/philox4x32_10_kat.txt)
and a uniformity test.
"""
from __future__ import annotations

import numpy as np

MASK32 = 0xFFFFFFFF
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
ROUNDS = 10


def _mulhilo(a: int, b: int):
    p = (a * b) & 0xFFFFFFFFFFFFFFFF
    return p >> 32, p & MASK32


def philox4x32_10(counter, key):
    """One Philox4x32-10 block: four 32-bit counter words, two key words -> four words."""
    c0, c1, c2, c3 = (int(x) & MASK32 for x in counter)
    k0, k1 = (int(x) & MASK32 for x in key)
    for r in range(ROUNDS):
        if r > 0:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        hi0, lo0 = _mulhilo(PHILOX_M0, c0)
        hi1, lo1 = _mulhilo(PHILOX_M1, c2)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def philox4x32_10_np(counter: np.ndarray, key: np.ndarray) -> np.ndarray:
    """Vectorised form of :func:`philox4x32_10`: counter uint [n,4], key uint [n,2]."""
    c = np.asarray(counter, dtype=np.uint64) & MASK32
    k = np.asarray(key, dtype=np.uint64) & MASK32
    c0, c1, c2, c3 = c[:, 0].copy(), c[:, 1].copy(), c[:, 2].copy(), c[:, 3].copy()
    k0, k1 = k[:, 0].copy(), k[:, 1].copy()
    m0, m1 = np.uint64(PHILOX_M0), np.uint64(PHILOX_M1)
    for r in range(ROUNDS):
        if r > 0:
            k0 = (k0 + np.uint64(PHILOX_W0)) & np.uint64(MASK32)
            k1 = (k1 + np.uint64(PHILOX_W1)) & np.uint64(MASK32)
        p0 = m0 * c0  # < 2^64: both factors are < 2^32
        p1 = m1 * c2
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(MASK32)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(MASK32)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return np.stack([c0, c1, c2, c3], axis=1).astype(np.uint32)


def uniform24(seed: int, step: int) -> float:
    """The sampler's uniform in [0, 1): 24 high bits of Philox word 0."""
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    step = int(step) & 0xFFFFFFFFFFFFFFFF
    x0 = philox4x32_10((step & MASK32, step >> 32, 0, 0), (seed & MASK32, seed >> 32))[0]
    return (x0 >> 8) * 2.0 ** -24


def uniform24_np(seeds: np.ndarray, step: int) -> np.ndarray:
    """Vectorised :func:`uniform24` over an array of uint64 seeds (one step)."""
    seeds = np.asarray(seeds, dtype=np.uint64).reshape(-1)
    n = seeds.size
    step = int(step) & 0xFFFFFFFFFFFFFFFF
    ctr = np.zeros((n, 4), dtype=np.uint64)
    ctr[:, 0] = step & MASK32
    ctr[:, 1] = step >> 32
    key = np.stack([seeds & np.uint64(MASK32), seeds >> np.uint64(32)], axis=1)
    x0 = philox4x32_10_np(ctr, key)[:, 0].astype(np.float64)
    return np.floor(x0 / 256.0) * 2.0 ** -24
