"""Pins of the residual-stream precheck oracle (App. A).

Anchors that do not go through the oracle's own formula: the logistic
function's closed-form values and symmetry, the library logistic routine as
a special case, a 3-d example computed by hand, and the extremes of the
threshold.
"""
import math

import numpy as np
import pytest

from oracle import gate as ogate
from oracle import precheck


def test_zero_weights_or_zero_activation_give_sigmoid_of_bias():
    rng = np.random.default_rng(0)
    h = rng.standard_normal((5, 16))
    for b in (-3.0, 0.0, 0.7):
        z, p, _ = precheck.precheck(h, np.zeros(16), b, 0.5)
        assert np.all(z == b)
        assert np.allclose(p, 1.0 / (1.0 + math.exp(-b)), rtol=0, atol=1e-15)
        z, p, _ = precheck.precheck(np.zeros((3, 16)), rng.standard_normal(16), b, 0.5)
        assert np.all(z == b)


def test_hand_computed_three_dim_case():
    # w = (1, -2, 0.5), h = (2, 1, 4), b = -1  ->  z = 2 - 2 + 2 - 1 = 1
    z, p, skip = precheck.precheck(np.array([[2.0, 1.0, 4.0]]), np.array([1.0, -2.0, 0.5]), -1.0, 0.5)
    assert z[0] == 1.0
    assert abs(p[0] - 0.7310585786300049) < 1e-15  # 1 / (1 + e^-1)
    assert not skip[0]
    _, _, skip = precheck.precheck(np.array([[2.0, 1.0, 4.0]]), np.array([1.0, -2.0, 0.5]), -1.0, 0.75)
    assert skip[0]


def test_sigmoid_symmetry_and_library_agreement():
    scipy_special = pytest.importorskip("scipy.special")
    z = np.concatenate([np.linspace(-40, 40, 801), [-745.0, -700.0, 700.0, 745.0]])
    p = precheck.sigmoid(z)
    assert np.all(np.isfinite(p)) and np.all((p >= 0) & (p <= 1))
    assert np.allclose(p + precheck.sigmoid(-z), 1.0, rtol=0, atol=1e-15)
    assert np.allclose(p, scipy_special.expit(z), rtol=1e-14, atol=1e-300)
    assert np.all(np.diff(p[:801]) >= 0)  # monotone


def test_threshold_extremes():
    rng = np.random.default_rng(1)
    h, w = rng.standard_normal((64, 32)), rng.standard_normal(32)
    _, p, skip = precheck.precheck(h, w, 0.0, 0.0)
    assert not np.any(skip & (p > 0))
    _, _, skip = precheck.precheck(h, w, 0.0, 1.0)
    assert np.all(skip)  # every probability is <= 1


def test_threshold_is_inclusive():
    # App. A skips when the predicted probability is at most theta: at z = 0 the
    # logistic is exactly 1/2, so theta = 1/2 skips and the next double below does not
    h, w = np.ones((2, 8)), np.zeros(8)
    z, p, skip = precheck.precheck(h, w, 0.0, 0.5)
    assert np.all(z == 0.0) and np.all(p == 0.5) and np.all(skip)
    _, _, skip = precheck.precheck(h, w, 0.0, np.nextafter(0.5, 0.0))
    assert not np.any(skip)


def test_apply_masks_only_skipped_fresh_groups():
    states = [ogate.GateState() for _ in range(4)]
    states[3].steps = 1  # a probe that already started is left alone
    active = np.ones(4 * 3, np.uint8)
    out = precheck.apply(states, np.array([True, False, True, True]), 3, active)
    assert [s.decision for s in states] == [ogate.NON_REFUSAL, ogate.PENDING, ogate.NON_REFUSAL, ogate.PENDING]
    assert [s.done for s in states] == [True, False, True, False]
    assert all(s.decisive_step == -1 for s in states)
    expect = np.ones(12, np.uint8)
    expect[[0, 6]] = 0  # probe rows of groups 0 and 2; their sample rows go on
    assert np.array_equal(out, expect)
    # masked rows stay masked, and the input array is not modified
    assert np.all(active == 1)
