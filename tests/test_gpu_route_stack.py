"""GPU parity of routing (Sec. 3.2, Eq. 13), the MLP stack and calibration."""
import numpy as np
import pytest
import torch

from paper_2607_08991_gb300 import inputs
from tests import _parity as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sats():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08991_gb300 import sats as s
    return s


# ---------------------------------------------------------------- routing

@pytest.mark.parametrize("B,V,p,zipf", [
    (1, 151936, 0.3, False), (8, 151936, 0.3, False), (64, 151936, 0.3, False),
    (256, 128256, 0.2, True), (2048, 128256, 0.2, True), (3001, 1000, 0.5, False),
    (1500, 50, 0.0, False), (1500, 50, 1.0, False),
])
def test_route_bit_exact(sats, oracle, B, V, p, zipf):
    lut = inputs.routing_lut(V, p, seed=inputs.SEED_LUT + B)
    ids = (inputs.token_ids_zipf(B, V, seed=inputs.SEED_IDS + B) if zipf
           else inputs.token_ids_uniform(B, V, seed=inputs.SEED_IDS + B))
    perm_ref, nd_ref = oracle.route(ids, lut)
    perm = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    nd = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    sats.route(P.dev(ids), P.dev(lut), perm, nd, st)
    assert sats.get_status_word(st) == sats.OK
    assert int(nd.item()) == nd_ref
    assert np.array_equal(perm.cpu().numpy(), perm_ref)


def test_route_bad_token_flags_status(sats):
    lut = np.zeros(10, np.uint8)
    ids = np.array([3, 10, -1, 4], np.int32)
    perm = torch.empty(4, dtype=torch.int32, device="cuda")
    nd = torch.empty(1, dtype=torch.int32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    sats.route(P.dev(ids), P.dev(lut), perm, nd, st)
    assert sats.get_status_word(st) == sats.EDEVICE
    # out-of-range ids take the base path, in order
    assert int(nd.item()) == 2 and perm.cpu().tolist() == [1, 2, 0, 3]
    assert sats.get_status_word(st) == sats.OK          # cleared by the read


# ---------------------------------------------------------------- stack

def _stack(sats, oracle, L, H, N, B, targets, eps, routed=False, V=1000, p_dense=0.3, seed=0):
    ws_ = [inputs.mlp_weights(H, N, layer=l, seed=inputs.SEED_WEIGHTS + 50 * seed) for l in range(L)]
    nw = [inputs.norm_weight(H, layer=l) for l in range(L)]
    x0 = inputs.activations_f32(B, H, seed=inputs.SEED_X + seed)
    # per-layer thresholds from the oracle's Eq. 3 on calibration vectors run through the stack
    cal = inputs.activations_f32(8, H, seed=inputs.SEED_CALIB).astype(np.float64)
    t = []
    for l in range(L):
        n = oracle.rmsnorm(cal, nw[l], eps)
        tl = float(np.float32(oracle.percentile_threshold(oracle.gate_act(n, ws_[l].Wg), targets[l])))
        t.append(tl)
        y, *_ = oracle.sparse_mlp(n, ws_[l].Wg, ws_[l].Wu, ws_[l].Wd, tl)
        cal = cal + y
    ids = lut = None
    if routed:
        lut = inputs.routing_lut(V, p_dense, seed=inputs.SEED_LUT + seed)
        ids = inputs.token_ids_uniform(B, V, seed=inputs.SEED_IDS + seed)
    layers = [sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd)) for w in ws_]
    ws = sats.Workspace(H, N, B)
    x = P.dev(x0.copy())
    trace = torch.full((L, B, N), 7, dtype=torch.uint8, device="cuda")
    sats.mlp_stack(layers, [P.dev(w) for w in nw], t, eps, x, ws,
                   token_ids=None if ids is None else P.dev(ids), lut=None if lut is None else P.dev(lut),
                   keep_trace=trace)
    assert sats.get_error(ws) == sats.OK
    keep_gpu = trace.cpu().numpy()
    assert set(np.unique(keep_gpu).tolist()) <= {0, 1}
    x_ref, keep_ref, nb = oracle.mlp_stack(x0.astype(np.float64), [w.Wg for w in ws_], [w.Wu for w in ws_],
                                           [w.Wd for w in ws_], nw, t, eps, ids=ids, lut=lut,
                                           keep_hint=keep_gpu, band_rel=P.BAND_REL, want_keep=True)
    assert np.array_equal(keep_gpu, keep_ref), "per-layer kept sets differ outside the band"
    P.assert_close(x.cpu().numpy(), x_ref)
    for l in layers:
        l.close()
    return keep_ref, ids, lut


@pytest.mark.parametrize("L,H,N,B", [
    (3, 256, 512, 1), (4, 512, 1408, 3), (2, 1024, 333, 6),
    (2, 8192, 200, 1),   # the largest hidden size: four vectors per decode-kernel thread, RMSNorm gains in registers
    (2, 8192, 200, 3),   # ... and on the tensor cores (one token per decode pass above 4096): the split kernel's full row
])
def test_stack_matches_oracle(sats, oracle, L, H, N, B):
    targets = inputs.stack_sparsity_targets(L, 0.55, 0.85)
    _stack(sats, oracle, L, H, N, B, targets, 1e-5)


@pytest.mark.parametrize("B", [1, 8, 64])
def test_routed_stack_matches_oracle(sats, oracle, B):
    L, H, N = 3, 512, 1408
    keep, ids, lut = _stack(sats, oracle, L, H, N, B, [0.5] * L, 1e-6, routed=True, p_dense=0.4, seed=B)
    dense = lut[ids] == 1
    assert keep[:, dense].all()


@pytest.mark.parametrize("B,p_dense", [(300, 0.4), (8, 1.0), (8, 0.0), (300, 1.0), (300, 0.0)])
def test_routed_stack_tensor_core_groups(sats, oracle, B, p_dense):
    """Batches on the tensor cores work in routed order (base-path tokens first, gathered
    by the routing permutation, results scattered back): a mixed batch beyond one 128-token
    tile, and the all-base / all-sparse tables, which must equal the static dense and sparse
    paths."""
    L, H, N = 2, 512, 1408
    keep, ids, lut = _stack(sats, oracle, L, H, N, B, [0.6] * L, 1e-6, routed=True, p_dense=p_dense, seed=B + 1)
    dense = lut[ids] == 1
    assert keep[:, dense].all()
    if p_dense == 1.0:
        assert keep.all()
    if p_dense == 0.0:
        assert abs((1.0 - keep.mean()) - 0.6) < 0.1


def test_llama_shaped_stack_two_layers(sats, oracle):
    """Two Llama-3.1-8B-shaped blocks (4096 / 14336), one decode token."""
    _stack(sats, oracle, 2, inputs.LLAMA_H, inputs.LLAMA_N, 1, [0.6, 0.8], 1e-5)


def test_stack_bad_token_reports_device_error(sats):
    H, N, B, V = 64, 64, 2, 16
    w = inputs.mlp_weights(H, N)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    x = P.dev(inputs.activations_f32(B, H))
    sats.mlp_stack([layer], [P.dev(inputs.norm_weight(H))], [0.1], 1e-5, x, ws,
                   token_ids=P.dev(np.array([1, 99], np.int32)), lut=P.dev(np.zeros(V, np.uint8)))
    assert sats.get_error(ws) == sats.EDEVICE
    assert sats.get_error(ws) == sats.OK


# ---------------------------------------------------------------- calibration

def test_gate_act_and_percentile(sats, oracle):
    H, N, C = 512, 1408, 64
    w = inputs.mlp_weights(H, N)
    xc = inputs.activations_bf16(C, H, seed=inputs.SEED_CALIB)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    a = torch.empty(C, N, dtype=torch.float32, device="cuda")
    sats.gate_act(layer, P.dev_u16(xc), a)
    a_ref = oracle.gate_act(oracle.bf16_to_f64(xc), w.Wg)
    a_gpu = a.cpu().numpy()
    np.testing.assert_allclose(a_gpu, a_ref, rtol=1e-4, atol=1e-5)
    sel = torch.empty(sats.select_workspace_bytes(), dtype=torch.uint8, device="cuda")
    for k in (0.1, 0.5, 0.7, 0.9, 1.0, 0.0, 1.5):
        t = sats.percentile_threshold(a, k, sel)
        # selection is exact: the same rule on the same fp32 values
        assert t == oracle.percentile_threshold(a_gpu.astype(np.float64), k), k
