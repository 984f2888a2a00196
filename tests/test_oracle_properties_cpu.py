"""Property tests (hypothesis, random small shapes and seeds) for the oracle.

Each property states the definition directly, element by element in Python
floats, and compares the oracle with it:
- the thresholded MLP (Sec. 2, Eqs. 1-5): g, a = SiLU(g), the mask |a| >= t,
  h = mask * a * u and y = h W_down, for any threshold drawn between the
  activations (neurons within 1e-9 of t are not compared);
- the percentile threshold (Eq. 3): the smallest magnitude t with
  #(|v| <= t) >= ceil(k n), so that #(|v| < t) < ceil(k n);
- routing (Eq. 13 as a LUT): the base-path tokens first, then the others, each
  group in increasing token order.
"""
import math

import numpy as np
import pytest

from paper_2607_08991_gb300 import inputs

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402


def _brute_mlp(x, Wg, Wu, Wd, t):
    B, H = x.shape
    N = Wg.shape[1]
    a = np.zeros((B, N))
    y = np.zeros((B, Wd.shape[1]))
    keep = np.zeros((B, N), dtype=bool)
    for b in range(B):
        h = [0.0] * N
        for j in range(N):
            g = math.fsum(x[b, k] * Wg[k, j] for k in range(H))
            u = math.fsum(x[b, k] * Wu[k, j] for k in range(H))
            a[b, j] = g / (1.0 + math.exp(-g))
            keep[b, j] = abs(a[b, j]) >= t
            h[j] = a[b, j] * u if keep[b, j] else 0.0
        for i in range(Wd.shape[1]):
            y[b, i] = math.fsum(h[j] * Wd[j, i] for j in range(N))
    return y, a, keep


@settings(max_examples=40, deadline=None)
@given(H=st.integers(1, 9), N=st.integers(1, 9), B=st.integers(1, 3), seed=st.integers(0, 10 ** 6),
       q=st.floats(0.0, 1.0))
def test_sparse_mlp_is_its_definition(oracle, H, N, B, seed, q):
    w = inputs.mlp_weights(H, N, std=0.5, seed=seed)
    x = oracle.bf16_to_f64(inputs.activations_bf16(B, H, seed=seed + 1))
    Wg, Wu, Wd = (oracle.bf16_to_f64(m) for m in (w.Wg, w.Wu, w.Wd))
    _, a_ref, _ = _brute_mlp(x, Wg, Wu, Wd, 0.0)
    mags = np.sort(np.abs(a_ref).ravel())
    t = float(mags[min(int(q * mags.size), mags.size - 1)]) * 0.999 + 1e-300
    y_ref, a_ref, keep_ref = _brute_mlp(x, Wg, Wu, Wd, t)
    y, a, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, t)
    np.testing.assert_allclose(a, a_ref, rtol=1e-12, atol=1e-300)
    far = np.abs(np.abs(a_ref) - t) > 1e-9 * t
    assert np.array_equal(keep.astype(bool)[far], keep_ref[far])
    if far.all():
        np.testing.assert_allclose(y, y_ref, rtol=1e-11, atol=1e-12 * (1.0 + np.abs(y_ref).max()))


@settings(max_examples=60, deadline=None)
@given(v=st.lists(st.floats(-1e3, 1e3, allow_nan=False), min_size=1, max_size=40),
       k=st.floats(0.01, 1.0))
def test_percentile_threshold_is_eq3(oracle, v, k):
    v = np.array(v)
    t = oracle.percentile_threshold(v, k)
    mags = np.abs(v)
    m = max(1, math.ceil(k * v.size - 1e-12))
    assert t in set(mags.tolist())
    assert np.count_nonzero(mags <= t) >= m
    assert np.count_nonzero(mags < t) < m


@settings(max_examples=60, deadline=None)
@given(lut=st.lists(st.integers(0, 1), min_size=1, max_size=50), data=st.data())
def test_route_is_a_stable_partition(oracle, lut, data):
    V = len(lut)
    ids = np.array(data.draw(st.lists(st.integers(0, V - 1), min_size=1, max_size=30)), dtype=np.int32)
    perm, nd = oracle.route(ids, np.array(lut, dtype=np.uint8))
    dense = [b for b in range(ids.size) if lut[ids[b]] == 1]
    sparse = [b for b in range(ids.size) if lut[ids[b]] == 0]
    assert nd == len(dense)
    assert perm.tolist() == dense + sparse
