"""Pins for the oracle's routing calibration (Sec. 3.2, Eqs. 11-14), by hand."""
import numpy as np
import pytest


def test_scores_by_hand(oracle):
    #           occurrence: 0    1    2    3    4    5
    ids = np.array([       2,   0,   2,   3,   2,   0])
    l_base = np.array([  1.0, 2.0, 1.5, 0.5, 3.0, 2.0])
    l_sparse = np.array([1.5, 1.0, 2.5, 0.5, 3.3, 2.4])
    # d = max(0, ls - lb):  0.5, 0, 1.0, 0, 0.3, 0.4
    s = oracle.token_scores(ids, l_base, l_sparse, V=5)
    assert s[0] == pytest.approx((0.0 + 0.4) / 2)
    assert s[2] == pytest.approx((0.5 + 1.0 + 0.3) / 3)
    assert s[3] == 0.0
    assert np.isinf(s[1]) and np.isinf(s[4])          # never seen: base path
    with pytest.raises(ValueError):
        oracle.token_scores([5], [0.0], [1.0], V=5)


def test_threshold_by_hand(oracle):
    score = np.array([0.2, np.inf, 0.6, 0.0, 0.2])
    held = np.array([0, 0, 2, 3, 4, 1, 2, 2])          # scores 0.2 0.2 0.6 0 0.2 inf 0.6 0.6
    # candidates: 0 (R 0), 0.2 (R 1/8: only the 0), 0.6 (R 4/8), inf (R 7/8)
    assert oracle.routed_fraction(score, held, 0.2) == 1 / 8
    assert oracle.routed_fraction(score, held, 0.6) == 4 / 8
    assert oracle.route_threshold(score, held, 0.5) == (0.6, 0.5)
    assert oracle.route_threshold(score, held, 0.9) == (np.inf, 7 / 8)
    assert oracle.route_threshold(score, held, 0.05) == (0.0, 0.0)
    # 0.3125 is equally far from 1/8 and 4/8: the smaller tau wins
    tau, R = oracle.route_threshold(score, held, 0.3125)
    assert (tau, R) == (0.2, 1 / 8)
    lut = oracle.route_lut(score, 0.6)
    assert lut.tolist() == [0, 1, 1, 0, 0]


def test_routed_fraction_is_monotone(oracle):
    rng = np.random.default_rng(3)
    score = rng.random(50)
    held = rng.integers(0, 50, 400)
    R = [oracle.routed_fraction(score, held, t) for t in np.linspace(0, 1.2, 30)]
    assert np.all(np.diff(R) >= 0) and R[0] == 0.0 and R[-1] == 1.0
