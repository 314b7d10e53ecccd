"""Pins of the oracle's greedy step and min-p / inverse-CDF sampler.

Each check is anchored outside the oracle's own formula: brute-force loops,
scipy's softmax, closed-form CDF examples, limits (T -> 0, p_min = 1) and the
empirical draw frequency over many Philox seeds.
"""
import numpy as np
import pytest

from oracle import sampling
from oracle.philox import uniform24_np
from paper_2607_20791_gb300 import workloads


def _brute_argmax(row):
    best, arg = -np.inf, -1
    for i, v in enumerate(row):
        if v > best:
            best, arg = v, i
    return arg


def test_greedy_lowest_index_on_ties():
    rng = np.random.default_rng(1)
    for _ in range(50):
        row = rng.integers(-5, 5, size=257).astype(np.float32)
        assert sampling.greedy_token(row) == _brute_argmax(row)
    row = np.zeros(10, np.float32)
    row[[3, 7]] = 2.0
    assert sampling.greedy_token(row) == 3


def test_greedy_on_bf16_ties():
    l32 = workloads.zipf_logits(4, 4096, seed=3)
    bits = workloads.f32_to_bf16_bits(l32)
    lb = sampling.bf16_bits_to_f32(bits)
    for r in range(4):
        assert sampling.greedy_token(lb[r]) == _brute_argmax(lb[r])


def test_bf16_decode_exact():
    # bit patterns decoded by hand: 0x3f80 = 1.0, 0xc020 = -2.5, 0x3e20 = 0.15625
    bits = np.array([0x3F80, 0xC020, 0x3E20, 0x0000, 0x8000], np.uint16)
    assert sampling.bf16_bits_to_f32(bits).tolist() == [1.0, -2.5, 0.15625, 0.0, -0.0]
    # exactly representable values survive the round trip
    y = np.array([1.0, -2.5, 0.15625, 96.0, 0.0], np.float32)
    assert np.array_equal(sampling.bf16_bits_to_f32(workloads.f32_to_bf16_bits(y)), y)


def test_min_p_set_matches_softmax_definition():
    scipy_special = pytest.importorskip("scipy.special")
    l32 = workloads.zipf_logits(8, 32000, seed=5)
    for r, (t, m) in enumerate([(1.0, 0.05), (1.5, 0.1), (2.0, 0.05), (3.0, 0.1),
                                (5.0, 0.3), (10.0, 0.05), (0.7, 0.2), (1.0, 0.0)]):
        row = l32[r]
        p = scipy_special.softmax(row.astype(np.float64) / t)
        exact = p >= m * p.max()
        kept = sampling.kept_set(row, t, m)
        margin = sampling.kept_set_margin(row, t, m)
        differ = kept != exact
        # the fp32 statement of the cutoff only differs from the exact set at
        # tokens within fp32 rounding of the threshold
        assert np.all(np.abs(margin[differ]) < 1e-5), (r, np.abs(margin[differ]).min())
        assert kept[int(np.argmax(row))]


def test_min_p_one_keeps_only_maxima():
    row = np.array([0.5, 2.0, 2.0, -1.0, 1.999], np.float32)
    kept = sampling.kept_set(row, 1.3, 1.0)
    assert kept.tolist() == [False, True, True, False, False]


def test_min_p_zero_keeps_all():
    row = np.array([-30.0, 0.0, 5.0, -np.float32(1e30)], np.float32)
    assert sampling.kept_set(row, 2.0, 0.0).all()


def test_inverse_cdf_closed_form():
    # logits ln(1..4), T = 1, no truncation: p = (1,2,3,4)/10; CDF 0.1 0.3 0.6 1.0
    row = np.log(np.array([1.0, 2.0, 3.0, 4.0])).astype(np.float32)
    for u, tok in [(0.0, 0), (0.05, 0), (0.15, 1), (0.29, 1), (0.31, 2), (0.59, 2),
                   (0.61, 3), (0.999, 3)]:
        assert sampling.sample_from_uniform(row, 1.0, 0.0, u).token == tok
    # T = 2 halves the log-odds: weights sqrt(1..4)
    w = np.sqrt([1.0, 2.0, 3.0, 4.0])
    cdf = np.cumsum(w) / w.sum()
    for u in [0.05, 0.2, 0.45, 0.7, 0.95]:
        expect = int(np.searchsorted(cdf, u, side="right"))
        assert sampling.sample_from_uniform(row, 2.0, 0.0, u).token == expect
    # min-p = 0.5 at T = 1 keeps p >= 0.2, i.e. tokens 1, 2, 3 with weights 2,3,4
    res = sampling.sample_from_uniform(row, 1.0, 0.5, 0.0)
    assert res.kept.tolist() == [False, True, True, True] and res.token == 1
    assert sampling.sample_from_uniform(row, 1.0, 0.5, 2.5 / 9).token == 2
    assert sampling.sample_from_uniform(row, 1.0, 0.5, 5.5 / 9).token == 3


def test_boundary_flag():
    row = np.log(np.array([1.0, 1.0, 2.0])).astype(np.float32)
    # CDF steps at 0.25, 0.5, 1.0
    assert sampling.sample_from_uniform(row, 1.0, 0.0, 0.25).boundary
    assert not sampling.sample_from_uniform(row, 1.0, 0.0, 0.3).boundary
    # the band is 1e-6 of Z on either side of a step: draws 5e-7 away are
    # flagged, draws 2e-6 away are not
    for du, flagged in ((5e-7, True), (-5e-7, True), (2e-6, False), (-2e-6, False)):
        for step in (0.25, 0.5):
            assert sampling.sample_from_uniform(row, 1.0, 0.0, step + du).boundary == flagged, (step, du)


def test_temperature_to_zero_is_greedy():
    l32 = workloads.zipf_logits(6, 4096, seed=9)
    for r in range(6):
        row = l32[r]
        assert np.sum(row == row.max()) == 1
        for u in [0.0, 0.3, 0.999]:
            assert sampling.sample_from_uniform(row, 1e-4, 0.0, u).token == int(np.argmax(row))
        res = sampling.sample_row(row, False, 0.0, 0.1, 123, 0)
        assert res.token == int(np.argmax(row))


def test_probe_rows_ignore_temperature():
    row = np.array([0.0, 3.0, 1.0], np.float32)
    assert sampling.sample_row(row, True, 5.0, 0.0, 1, 1).token == 1
    # 64 nearly equal logits: a T = 5 draw lands on the maximum ~1.7 % of the
    # time, a probe row (G_M, greedy) always does
    row = np.zeros(64, np.float32)
    row[17] = 0.5
    for seed in range(20):
        assert sampling.sample_row(row, True, 5.0, 0.0, seed, 1).token == 17
        assert sampling.sample_row(row, True, 5.0, 0.3, seed, 1).kept is None


def test_draw_frequencies_match_weights():
    scipy_stats = pytest.importorskip("scipy.stats")
    row = np.log(np.array([0.1, 0.2, 0.3, 0.4])).astype(np.float32)
    n = 40_000
    seeds = np.arange(n, dtype=np.uint64) * np.uint64(2654435761) + np.uint64(12345)
    toks = np.array([sampling.sample_row(row, False, 1.0, 0.0, int(s), 0).token for s in seeds])
    counts = np.bincount(toks, minlength=4)
    chi2, p = scipy_stats.chisquare(counts, n * np.array([0.1, 0.2, 0.3, 0.4]))
    assert p > 1e-4


def test_sample_head_masks_inactive_rows():
    case = workloads.head_sweep(8, 4096, "f32", seed=2)
    active = np.array([1, 0, 1, 1, 0, 1, 1, 1], np.uint8)
    res = sampling.sample_head(case.logits, case.dtype, case.is_probe, case.temperature,
                               case.min_p, case.seed, case.step, active)
    assert res.tokens[1] == -1 and res.tokens[4] == -1
    assert all(res.tokens[i] >= 0 for i in range(8) if active[i])
