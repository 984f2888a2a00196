"""The library's host implementation of Eqs. 7-10 (sats_sats_select) against the
oracle's on the same candidate tables: both must make identical choices (the
comparisons involve no arithmetic beyond a mean of the chosen sparsities)."""
import numpy as np
import pytest


@pytest.fixture(scope="module")
def sats():
    from paper_2607_08991_gb300 import build
    build.build_library()
    from paper_2607_08991_gb300 import sats as s
    return s


def _same(sats, oracle, t, err, sp, s_tar, guard=-1, gt=0.0, gs=0.0):
    b1, t1, S1 = sats.sats_select(t, err, sp, s_tar, guard, gt, gs)
    b2, t2, S2 = oracle.sats_select(np.asarray(t), np.asarray(err), np.asarray(sp), s_tar, guard, gt, gs)
    assert b1 == b2
    np.testing.assert_array_equal(np.asarray(t1), t2)
    assert S1 == pytest.approx(S2, abs=1e-15)


def test_worked_table(sats, oracle):
    t = [[0.1, 0.2, 0.3], [0.1, 0.2, 0.3]]
    err = [[0.01, 0.05, 0.2], [0.02, 0.03, 0.1]]
    sp = [[0.3, 0.5, 0.7], [0.2, 0.6, 0.8]]
    for s_tar in (0.0, 0.1, 0.44, 0.52, 0.71, 1.0):
        _same(sats, oracle, t, err, sp, s_tar)
    _same(sats, oracle, t, err, sp, 0.5, guard=1, gt=0.25, gs=0.7)


def test_random_tables(sats, oracle):
    rng = np.random.default_rng(17)
    for trial in range(200):
        L, K = int(rng.integers(1, 6)), int(rng.integers(1, 8))
        t = rng.random((L, K)) * (rng.random() < 0.5 and 1.0 or 0.01)
        if trial % 7 == 0:
            t[:, 0] = t[:, -1]                  # repeated thresholds
        err = np.round(rng.random((L, K)) * 0.2, 2 if trial % 3 == 0 else 12)   # ties in the budgets
        sp = rng.random((L, K))
        guard = int(rng.integers(-1, L)) if L > 1 else -1
        _same(sats, oracle, t.tolist(), err.tolist(), sp.tolist(), float(rng.random()), guard, 0.3, 0.6)


def test_select_rejects_bad_arguments(sats):
    with pytest.raises(sats.SatsError):
        sats.sats_select([[float("nan")]], [[0.1]], [[0.5]], 0.5)
    with pytest.raises(sats.SatsError):
        sats.sats_select([[0.1]], [[0.1]], [[0.5]], 0.5, guard=3)
