"""Pins for the oracle's routing (Sec. 3.2, Eq. 13), RMSNorm and the block stack."""
import numpy as np
import pytest
import scipy.special

from paper_2607_08991_gb300 import inputs


def _f(bits):
    return inputs.bf16_bits_to_f32(bits).astype(np.float64)


# ---------------------------------------------------------------- routing

def _brute_route(ids, lut):
    order = sorted(range(len(ids)), key=lambda b: (0 if lut[ids[b]] else 1, b))
    return order, sum(1 for b in range(len(ids)) if lut[ids[b]])


@pytest.mark.parametrize("B", [0, 1, 2, 17, 64, 300])
def test_route_brute_force(oracle, B):
    V = 97
    lut = inputs.routing_lut(V, 0.3, seed=B + 1)
    ids = inputs.token_ids_uniform(B, V, seed=B + 2)
    perm, nd = oracle.route(ids, lut)
    order, nd_b = _brute_route(ids.tolist(), lut.tolist())
    assert perm.tolist() == order and nd == nd_b
    assert sorted(perm.tolist()) == list(range(B))        # a permutation


def test_route_all_dense_all_sparse_identity(oracle):
    V, B = 50, 33
    ids = inputs.token_ids_uniform(B, V, seed=3)
    perm, nd = oracle.route(ids, np.ones(V, np.uint8))
    assert perm.tolist() == list(range(B)) and nd == B
    perm, nd = oracle.route(ids, np.zeros(V, np.uint8))
    assert perm.tolist() == list(range(B)) and nd == 0


def test_route_rejects_out_of_range(oracle):
    lut = np.ones(10, np.uint8)
    for bad in ([0, 10], [-1], [3, 2**31 - 1]):
        with pytest.raises(ValueError):
            oracle.route(np.array(bad, np.int32), lut)


# ---------------------------------------------------------------- RMSNorm

def test_rmsnorm_closed_forms(oracle):
    H = 16
    w = inputs.norm_weight(H, seed=1)
    c = 3.0
    out = oracle.rmsnorm(np.full((1, H), c), w, 1e-5)
    np.testing.assert_allclose(out[0], c / np.sqrt(c * c + 1e-5) * w.astype(np.float64), rtol=1e-14)
    x = np.random.default_rng(2).standard_normal((3, H))
    o1 = oracle.rmsnorm(x, w, 0.0)
    o2 = oracle.rmsnorm(7.5 * x, w, 0.0)                     # scale invariance with eps = 0
    np.testing.assert_allclose(o1, o2, rtol=1e-13)
    np.testing.assert_allclose(np.sqrt(np.mean((o1 / w) ** 2, axis=1)), 1.0, rtol=1e-13)


# ---------------------------------------------------------------- stack

def _stack_inputs(L, H, N, B, seed=0):
    ws = [inputs.mlp_weights(H, N, layer=l, seed=100 + seed) for l in range(L)]
    nw = [inputs.norm_weight(H, layer=l, seed=200 + seed) for l in range(L)]
    x = inputs.activations_f32(B, H, seed=300 + seed).astype(np.float64)
    return ws, nw, x


def _numpy_dense_stack(x, ws, nw, eps):
    x = x.copy()
    for w, g in zip(ws, nw):
        n = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + eps) * g.astype(np.float64)
        gg = n @ _f(w.Wg)
        x = x + (gg * scipy.special.expit(gg) * (n @ _f(w.Wu))) @ _f(w.Wd)
    return x


def _run(oracle, x, ws, nw, t, eps, **kw):
    return oracle.mlp_stack(x, [w.Wg for w in ws], [w.Wu for w in ws], [w.Wd for w in ws], nw, t, eps, **kw)


def test_stack_threshold_zero_equals_dense_stack(oracle):
    L, H, N, B = 3, 16, 32, 2
    ws, nw, x = _stack_inputs(L, H, N, B)
    out, keep, _ = _run(oracle, x, ws, nw, np.zeros(L), 1e-5, want_keep=True)
    assert keep.all()
    np.testing.assert_allclose(out, _numpy_dense_stack(x, ws, nw, 1e-5), rtol=1e-11, atol=1e-12)
    V = 7
    ids = np.arange(B, dtype=np.int32)
    out_d, keep_d, _ = _run(oracle, x, ws, nw, np.full(L, 0.3), 1e-5, ids=ids, lut=np.ones(V, np.uint8),
                            want_keep=True)
    assert keep_d.all()
    np.testing.assert_allclose(out_d, out, rtol=1e-12, atol=1e-13)


def test_stack_threshold_inf_is_identity(oracle):
    L, H, N, B = 2, 8, 16, 3
    ws, nw, x = _stack_inputs(L, H, N, B, seed=1)
    out, keep, _ = _run(oracle, x, ws, nw, np.full(L, np.inf), 1e-6, want_keep=True)
    assert not keep.any()
    assert np.array_equal(out, x)


def test_stack_one_layer_is_norm_then_layer(oracle):
    H, N, B = 16, 24, 2
    ws, nw, x = _stack_inputs(1, H, N, B, seed=2)
    t = 0.05
    out, keep, _ = _run(oracle, x, ws, nw, [t], 1e-5, want_keep=True)
    n = oracle.rmsnorm(x, nw[0], 1e-5)
    y, _, k1, _ = oracle.sparse_mlp(n, ws[0].Wg, ws[0].Wu, ws[0].Wd, t)
    assert np.array_equal(keep[0], k1)
    np.testing.assert_allclose(out, x + y, rtol=1e-13, atol=1e-14)


def test_stack_routing_mixes_paths_per_token(oracle):
    L, H, N, B, V = 3, 16, 32, 4, 11
    ws, nw, x = _stack_inputs(L, H, N, B, seed=3)
    lut = np.zeros(V, np.uint8)
    lut[[2, 5]] = 1
    ids = np.array([5, 1, 2, 9], np.int32)                 # tokens 0 and 2 take the base path
    t = np.array([0.05, 0.1, 0.07])
    out, keep, _ = _run(oracle, x, ws, nw, t, 1e-5, ids=ids, lut=lut, want_keep=True)
    dense_out, _, _ = _run(oracle, x[[0, 2]], ws, nw, np.zeros(L), 1e-5)
    sparse_out, sk, _ = _run(oracle, x[[1, 3]], ws, nw, t, 1e-5, want_keep=True)
    np.testing.assert_allclose(out[[0, 2]], dense_out, rtol=1e-12, atol=1e-13)
    assert np.array_equal(out[[1, 3]], sparse_out)
    assert keep[:, [0, 2]].all() and np.array_equal(keep[:, [1, 3]], sk)
    with pytest.raises(ValueError):
        _run(oracle, x, ws, nw, t, 1e-5, ids=np.array([0, 1, 2, V], np.int32), lut=lut)
