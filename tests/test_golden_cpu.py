"""The oracle against its stored fixture (tests/golden/sparse_mlp_h16_n24_b2.txt).

The paper prints no worked example, so the fixture was written by the committed
script tests/golden/make_golden.py from the oracle alone (Sec. 2, Eqs. 1-5 at
the Eq. 3 threshold).  It guards the oracle against accidental change: the
threshold, the activations and y to within a few ulps (libm's exp may differ
between hosts), the keep masks exactly (no activation lies near the threshold).
"""
import importlib.util
import os

import numpy as np

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _fixture():
    vals = {}
    with open(os.path.join(GOLDEN, "sparse_mlp_h16_n24_b2.txt")) as f:
        for ln in f:
            if ln.startswith("#") or not ln.strip():
                continue
            key, rest = ln.split(" ", 1)
            vals[key] = rest.strip()
    return vals


def _case():
    spec = importlib.util.spec_from_file_location("make_golden", os.path.join(GOLDEN, "make_golden.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_oracle_matches_stored_fixture(oracle):
    g = _fixture()
    mk = _case()
    w, xb, cal = mk.case()
    t = oracle.percentile_threshold(oracle.gate_act(oracle.bf16_to_f64(cal), w.Wg), mk.K)
    y, a, keep, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, t)
    t_ref = float(g["t"])
    assert abs(t - t_ref) <= 1e-13 * abs(t_ref)
    for b in range(mk.B):
        a_ref = np.array([float(v) for v in g["a%d" % b].split()])
        y_ref = np.array([float(v) for v in g["y%d" % b].split()])
        keep_ref = np.array([c == "1" for c in g["keep%d" % b]])
        # the masks are compared exactly only because no activation is near the threshold
        assert np.min(np.abs(np.abs(a_ref) - t_ref)) > 1e-9 * t_ref
        np.testing.assert_allclose(a[b], a_ref, rtol=1e-13, atol=1e-15)
        assert np.array_equal(keep[b].astype(bool), keep_ref)
        np.testing.assert_allclose(y[b], y_ref, rtol=1e-12, atol=1e-14)
        assert 0 < keep_ref.sum() < mk.N
