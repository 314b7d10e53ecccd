"""Pins of the oracle's Philox4x32-10 against the published known-answer vectors."""
import os

import numpy as np
import pytest

from oracle import philox

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((tuple(w[0:4]), tuple(w[4:6]), tuple(w[6:10])))
    return rows


def test_known_answer_vectors_scalar():
    kat = _kat()
    assert len(kat) == 3
    for ctr, key, out in kat:
        assert philox.philox4x32_10(ctr, key) == out


def test_known_answer_vectors_vectorised():
    kat = _kat()
    ctr = np.array([k[0] for k in kat], dtype=np.uint64)
    key = np.array([k[1] for k in kat], dtype=np.uint64)
    out = philox.philox4x32_10_np(ctr, key)
    assert [tuple(int(x) for x in r) for r in out] == [k[2] for k in kat]


def test_vectorised_matches_scalar_random_blocks():
    rng = np.random.default_rng(0)
    ctr = rng.integers(0, 2**32, size=(64, 4), dtype=np.uint64)
    key = rng.integers(0, 2**32, size=(64, 2), dtype=np.uint64)
    out = philox.philox4x32_10_np(ctr, key)
    for i in range(64):
        assert tuple(int(x) for x in out[i]) == philox.philox4x32_10(ctr[i], key[i])


def test_uniform_is_24_bit_and_in_range():
    seeds = np.arange(1000, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15)
    u = philox.uniform24_np(seeds, 7)
    assert np.all(u >= 0.0) and np.all(u < 1.0)
    assert np.all(u * 2**24 == np.floor(u * 2**24))
    assert np.all(u.astype(np.float32).astype(np.float64) == u)
    for i in range(0, 1000, 97):
        assert philox.uniform24(int(seeds[i]), 7) == u[i]


def test_uniform_key_and_counter_mapping():
    # key = (seed lo, seed hi), counter = (step lo, step hi, 0, 0), word 0 >> 8
    seed, step = 0x0123456789ABCDEF, 0x1111222233334444
    x0 = philox.philox4x32_10((0x33334444, 0x11112222, 0, 0), (0x89ABCDEF, 0x01234567))[0]
    assert philox.uniform24(seed, step) == (x0 >> 8) / 2**24


def test_uniformity_chi_square():
    scipy_stats = pytest.importorskip("scipy.stats")
    seeds = np.arange(1 << 16, dtype=np.uint64)
    u = philox.uniform24_np(seeds, 3)
    counts, _ = np.histogram(u, bins=64, range=(0.0, 1.0))
    chi2 = float(((counts - counts.mean()) ** 2 / counts.mean()).sum())
    p = 1.0 - scipy_stats.chi2.cdf(chi2, df=63)
    assert p > 1e-4
