"""Pins for the oracle's thresholded gated MLP (Sec. 2, Eqs. 1-5) and Eq. 3.

Each test fixes the oracle to something other than itself: a closed form,
a library routine the definition reduces to, brute force on tiny inputs,
or an invariant that a dropped term, a wrong sign, index or transposed
operand would break.
"""
import math

import numpy as np
import pytest
import scipy.special

from paper_2607_08991_gb300 import inputs


def _layer(H, N, seed=11, std=0.02):
    return inputs.mlp_weights(H, N, layer=0, std=std, seed=seed)


def _f(bits):
    return inputs.bf16_bits_to_f32(bits).astype(np.float64)


# ---------------------------------------------------------------- SiLU (Eq. 2)

def test_silu_minimum_is_lambert_w(oracle):
    # SiLU attains its minimum -W(1/e) at z* = -1 - W(1/e) (W = Lambert W).
    w = float(scipy.special.lambertw(math.exp(-1.0)).real)
    zstar = -1.0 - w
    assert oracle.silu(zstar) == pytest.approx(-w, rel=1e-14)
    # and it is a minimum: neighbours are larger
    assert oracle.silu(zstar - 1e-4) > oracle.silu(zstar)
    assert oracle.silu(zstar + 1e-4) > oracle.silu(zstar)


def test_silu_tail_and_symmetry(oracle):
    for z in [0.0, 0.3, 1.0, 2.5, 7.0]:
        # z*sigmoid(z) - (-z)*sigmoid(-z) = z
        assert oracle.silu(z) - oracle.silu(-z) == pytest.approx(z, abs=1e-15)
        # library logistic
        assert oracle.silu(z) == pytest.approx(z * scipy.special.expit(z), rel=1e-15, abs=1e-300)
    assert oracle.silu(0.0) == 0.0
    assert oracle.silu(30.0) == pytest.approx(30.0, rel=1e-12)       # sigmoid -> 1
    assert abs(oracle.silu(-30.0)) < 1e-11                              # sigmoid -> 0


# ---------------------------------------------------------------- gate / up (Eq. 1)

def test_gate_act_brute_force_tiny(oracle):
    H, N, B = 3, 5, 2
    w = _layer(H, N, seed=5, std=0.7)
    x = np.array([[0.5, -1.25, 2.0], [1.0, 0.0, -0.75]])
    a = oracle.gate_act(x, w.Wg)
    Wg = _f(w.Wg)
    for b in range(B):
        for j in range(N):
            g = sum(x[b][k] * Wg[k][j] for k in range(H))
            assert a[b][j] == pytest.approx(g / (1.0 + math.exp(-g)), rel=1e-14, abs=1e-300)


def test_gate_and_up_match_numpy_nonsquare(oracle):
    H, N, B = 24, 40, 3
    w = _layer(H, N)
    x = np.random.default_rng(1).standard_normal((B, H))
    g = x @ _f(w.Wg)
    np.testing.assert_allclose(oracle.gate_act(x, w.Wg), g * scipy.special.expit(g), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(oracle.up_proj(x, w.Wu), x @ _f(w.Wu), rtol=1e-12, atol=1e-15)


def test_bf16_decode_exact(oracle):
    bits = np.array([0x0000, 0x8000, 0x3F80, 0xBF80, 0x4049, 0x3C23, 0x7F7F, 0x0001], dtype=np.uint16)
    want = [0.0, -0.0, 1.0, -1.0, 3.140625, 163.0 / 16384.0, 3.3895313892515355e38, 2.0 ** -133]
    got = oracle.bf16_to_f64(bits)
    for g, w_ in zip(got, want):
        assert g == pytest.approx(w_, rel=1e-12, abs=0)


# ---------------------------------------------------------------- mask (Eqs. 4-5)

def test_mask_brute_force_and_tie(oracle):
    H, N, B = 8, 16, 3
    w = _layer(H, N, seed=3, std=0.5)
    x = np.random.default_rng(2).standard_normal((B, H))
    a = oracle.gate_act(x, w.Wg)
    t = np.array([0.1, 0.25, 0.6])
    keep, nb = oracle.cats_mask(a, t)
    assert nb == 0
    for b in range(B):
        for j in range(N):
            assert keep[b][j] == (1 if abs(a[b][j]) >= t[b] else 0)
    # a magnitude exactly equal to t is kept (>=, Eq. 4)
    t_tie = np.abs(a[:, 7]).copy()
    keep2, _ = oracle.cats_mask(a, t_tie)
    assert keep2[:, 7].tolist() == [1, 1, 1]


def test_band_hint_only_inside_band(oracle):
    H, N, B = 8, 64, 2
    w = _layer(H, N, seed=4, std=0.5)
    x = np.random.default_rng(3).standard_normal((B, H))
    a = oracle.gate_act(x, w.Wg)
    t = np.array([0.3, 0.3])
    own, _ = oracle.cats_mask(a, t)
    flipped = (1 - own).astype(np.uint8)
    same, nb0 = oracle.cats_mask(a, t, keep_hint=flipped, band_rel=0.0)
    assert nb0 == 0 and np.array_equal(same, own)
    allband, nb = oracle.cats_mask(a, t, keep_hint=flipped, band_rel=1e9)
    assert nb == B * N and np.array_equal(allband, flipped)
    band = 0.2
    part, nbp = oracle.cats_mask(a, t, keep_hint=flipped, band_rel=band)
    inb = np.abs(np.abs(a) - t[:, None]) <= band * t[:, None]
    assert nbp == int(inb.sum())
    assert np.array_equal(part[inb], flipped[inb]) and np.array_equal(part[~inb], own[~inb])


# ---------------------------------------------------------------- full MLP

def _numpy_dense(x, w):
    g = x @ _f(w.Wg)
    h = g * scipy.special.expit(g) * (x @ _f(w.Wu))
    return h @ _f(w.Wd)


def test_threshold_zero_is_dense(oracle):
    H, N, B = 32, 48, 3
    w = _layer(H, N)
    x = np.random.default_rng(4).standard_normal((B, H))
    y, a, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, 0.0)
    assert keep.all()
    yd = oracle.dense_mlp(x, w.Wg, w.Wu, w.Wd)
    np.testing.assert_allclose(y, yd, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(yd, _numpy_dense(x, w), rtol=1e-11, atol=1e-14)


def test_threshold_inf_is_zero(oracle):
    H, N, B = 16, 24, 2
    w = _layer(H, N)
    x = np.random.default_rng(5).standard_normal((B, H))
    y, a, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, np.inf)
    assert not keep.any()
    assert np.all(y == 0.0)


def test_masked_matches_numpy(oracle):
    H, N, B = 24, 56, 4
    w = _layer(H, N)
    x = np.random.default_rng(6).standard_normal((B, H))
    t = np.array([0.0, 0.05, 0.1, 0.2])
    y, a, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, t)
    g = x @ _f(w.Wg)
    act = g * scipy.special.expit(g)
    np.testing.assert_allclose(a, act, rtol=1e-12, atol=1e-15)
    m = np.abs(act) >= t[:, None]
    assert np.array_equal(keep.astype(bool), m)
    want = (np.where(m, act, 0.0) * (x @ _f(w.Wu))) @ _f(w.Wd)
    np.testing.assert_allclose(y, want, rtol=1e-11, atol=1e-14)
    assert 0 < keep[1:].sum() < (B - 1) * N


def test_skipped_neurons_are_never_used(oracle):
    H, N, B = 16, 40, 1
    w = _layer(H, N)
    x = np.random.default_rng(7).standard_normal((B, H))
    t = 0.08
    y, a, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, t)
    off = np.where(keep[0] == 0)[0]
    assert off.size > 0
    rng = np.random.default_rng(8)
    Wu2, Wd2 = w.Wu.copy(), w.Wd.copy()
    Wu2[:, off] = inputs.to_bf16_bits(rng.standard_normal((H, off.size)).astype(np.float32))
    Wd2[off, :] = inputs.to_bf16_bits(rng.standard_normal((off.size, H)).astype(np.float32))
    y2, _, keep2, _ = oracle.sparse_mlp(x, w.Wg, Wu2, Wd2, t)
    assert np.array_equal(keep, keep2)
    assert np.array_equal(y, y2)


def test_down_projection_linear(oracle):
    H, N = 16, 24
    w = _layer(H, N)
    x = np.random.default_rng(9).standard_normal((2, H))
    y, *_ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, 0.05)
    # doubling a bf16 value adds one to its exponent: exact
    Wd2 = inputs.to_bf16_bits(2.0 * inputs.bf16_bits_to_f32(w.Wd))
    y2, *_ = oracle.sparse_mlp(x, w.Wg, w.Wu, Wd2, 0.05)
    assert np.array_equal(y2, 2.0 * y)


def test_single_neuron_closed_form(oracle):
    wg, wu, wd = 0.75, -1.5, 0.5
    bits = lambda v: inputs.to_bf16_bits(np.array([[v]], dtype=np.float32))
    for x in [-2.0, -0.5, 0.25, 1.0, 3.0]:
        for t in [0.0, 0.2, 1.0]:
            y, a, keep, _ = oracle.sparse_mlp(np.array([[x]]), bits(wg), bits(wu), bits(wd), t)
            g = x * wg
            act = g / (1 + math.exp(-g))
            want = (act if abs(act) >= t else 0.0) * (x * wu) * wd
            assert y[0, 0] == pytest.approx(want, rel=1e-14, abs=1e-300)


def test_neuron_permutation_invariance(oracle):
    H, N = 16, 32
    w = _layer(H, N)
    x = np.random.default_rng(10).standard_normal((2, H))
    y, _, keep, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, 0.05)
    p = np.random.default_rng(11).permutation(N)
    y2, _, keep2, _ = oracle.sparse_mlp(x, w.Wg[:, p], w.Wu[:, p], w.Wd[p, :], 0.05)
    assert np.array_equal(keep2, keep[:, p])
    np.testing.assert_allclose(y2, y, rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- Eq. 3

@pytest.mark.parametrize("n", [1, 7, 100, 1000])
@pytest.mark.parametrize("k", [0.1, 0.25, 0.5, 0.7, 0.9, 1.0])
def test_percentile_matches_numpy_inverted_cdf(oracle, n, k):
    v = np.random.default_rng(n).standard_normal(n)
    t = oracle.percentile_threshold(v, k)
    assert t == np.percentile(np.abs(v), 100.0 * k, method="inverted_cdf")


def test_percentile_realised_sparsity_exact(oracle):
    v = np.random.default_rng(12).standard_normal(64 * 1408)
    n = v.size
    for k in [0.5, 0.7, 0.9, 0.3]:
        t = oracle.percentile_threshold(v, k)
        m = math.ceil(k * n - 1e-9)
        assert int((np.abs(v) < t).sum()) == m - 1
        assert int((np.abs(v) <= t).sum()) == m


def test_percentile_edges(oracle):
    v = np.array([3.0, -1.0, 2.0])
    assert oracle.percentile_threshold(v, 0.0) == 0.0
    assert oracle.percentile_threshold(v, 1.0) == 3.0
    assert oracle.percentile_threshold(v, 1.5) == math.inf
    assert oracle.percentile_threshold(v, 1.0 / 3.0) == 1.0
    assert oracle.percentile_threshold(v, 0.34) == 2.0
    # k*n = 0.3*10 must not round up to 4
    assert oracle.percentile_threshold(np.arange(1.0, 11.0), 0.3) == 3.0
