"""Pins for the oracle's LoRA sparse path (Sec. 4, fine-tuned routing: the sparse
path runs the thresholded MLP of Sec. 2, Eqs. 1-5, on adapted weights W + s A B).

The oracle applies each low-rank term factor by factor.  It is pinned against
(1) the same MLP on the merged weights W + s A B formed here in fp64 (numpy,
a different association of the same products: a dropped, transposed or
misplaced factor fails it); (2) the base oracle at s = 0; (3) the invariance
under A -> 2A, B -> B/2 (exact in bf16); (4) a closed form: with only the down
adapter, y - y_base = s (h A_d) B_d for the base mask and h.
"""
import numpy as np
import pytest

from paper_2607_08991_gb300 import inputs


def _setup(H, N, B, r, seed=1):
    w = inputs.mlp_weights(H, N, std=0.1, seed=seed)
    lo = inputs.lora_adapter(H, N, r, std_a=0.1, std_b=0.1, seed=seed + 11)
    x = inputs.activations_f32(B, H, seed=seed + 3).astype(np.float64)
    return w, lo, x


def _f(bits):
    return inputs.bf16_bits_to_f32(bits).astype(np.float64)


def _merged_reference(x, w, lo, s, t):
    """The thresholded MLP on merged fp64 weights W + s A B (Sec. 2, Eqs. 1-5)."""
    Ag, Bg, Au, Bu, Ad, Bd = (_f(m) for m in lo)
    Wg = _f(w.Wg) + s * Ag @ Bg
    Wu = _f(w.Wu) + s * Au @ Bu
    Wd = _f(w.Wd) + s * Ad @ Bd
    g = x @ Wg
    a = g / (1.0 + np.exp(-g))
    keep = np.abs(a) >= t
    h = np.where(keep, a * (x @ Wu), 0.0)
    return h @ Wd, a, keep


def _gap_threshold(a, q=0.5):
    v = np.sort(np.abs(a).ravel())
    i = int(q * (v.size - 1))
    while v[i + 1] - v[i] < 1e-6 * v[i + 1]:
        i += 1
    return 0.5 * (v[i] + v[i + 1])


@pytest.mark.parametrize("H,N,B,r,s", [(16, 24, 3, 4, 0.5), (32, 40, 2, 8, 2.0), (8, 8, 1, 1, 1.0)])
def test_lora_equals_merged_weights(oracle, H, N, B, r, s):
    w, lo, x = _setup(H, N, B, r)
    _, a_m, _ = _merged_reference(x, w, lo, s, 0.0)
    t = _gap_threshold(a_m)
    y_ref, a_ref, keep_ref = _merged_reference(x, w, lo, s, t)
    y, a, keep, _ = oracle.sparse_mlp_lora(x, w.Wg, w.Wu, w.Wd, lo, s, t)
    np.testing.assert_allclose(a, a_ref, rtol=1e-12, atol=1e-14)
    assert np.array_equal(keep.astype(bool), keep_ref)
    assert 0 < keep.sum() < keep.size
    np.testing.assert_allclose(y, y_ref, rtol=1e-11, atol=1e-13)


def test_lora_scale_zero_is_the_base_mlp(oracle):
    H, N, B, r = 24, 36, 3, 4
    w, lo, x = _setup(H, N, B, r, seed=5)
    t = _gap_threshold(oracle.gate_act(x, w.Wg))
    y0, a0, k0, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, t)
    y1, a1, k1, _ = oracle.sparse_mlp_lora(x, w.Wg, w.Wu, w.Wd, lo, 0.0, t)
    assert np.array_equal(k0, k1)
    np.testing.assert_allclose(a1, a0, rtol=1e-13, atol=0)
    np.testing.assert_allclose(y1, y0, rtol=1e-12, atol=1e-15)


def test_lora_factor_rescaling_is_invariant(oracle):
    H, N, B, r = 16, 20, 2, 3
    w, lo, x = _setup(H, N, B, r, seed=9)
    t = 0.05

    def times2(bits):   # x 2 exactly: add one to the bf16 exponent of the non-zero values
        out = bits.copy()
        nz = (out & 0x7FFF) != 0
        out[nz] = out[nz] + 0x0080
        return out

    def half(bits):
        out = bits.copy()
        nz = (out & 0x7FFF) != 0
        out[nz] = out[nz] - 0x0080
        return out

    Ag, Bg, Au, Bu, Ad, Bd = lo
    lo2 = (times2(Ag), half(Bg), times2(Au), half(Bu), times2(Ad), half(Bd))
    y1, a1, k1, _ = oracle.sparse_mlp_lora(x, w.Wg, w.Wu, w.Wd, lo, 1.5, t)
    y2, a2, k2, _ = oracle.sparse_mlp_lora(x, w.Wg, w.Wu, w.Wd, lo2, 1.5, t)
    assert np.array_equal(k1, k2)
    np.testing.assert_allclose(a2, a1, rtol=1e-14)
    np.testing.assert_allclose(y2, y1, rtol=1e-13, atol=1e-16)


def test_lora_down_adapter_alone_closed_form(oracle):
    """B_g = B_u = 0: mask and h are the base ones; y moves by exactly s (h A_d) B_d."""
    H, N, B, r, s = 20, 30, 3, 5, 0.75
    w, lo, x = _setup(H, N, B, r, seed=13)
    Ag, Bg, Au, Bu, Ad, Bd = lo
    lo_d = (Ag, np.zeros_like(Bg), Au, np.zeros_like(Bu), Ad, Bd)
    t = _gap_threshold(oracle.gate_act(x, w.Wg))
    y0, a0, k0, _ = oracle.sparse_mlp(x, w.Wg, w.Wu, w.Wd, t)
    y1, a1, k1, _ = oracle.sparse_mlp_lora(x, w.Wg, w.Wu, w.Wd, lo_d, s, t)
    assert np.array_equal(k0, k1)
    h = np.where(k0.astype(bool), a0 * oracle.up_proj(x, w.Wu), 0.0)
    np.testing.assert_allclose(y1 - y0, s * (h @ _f(Ad)) @ _f(Bd), rtol=1e-9, atol=1e-12)
