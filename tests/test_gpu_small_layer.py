"""GPU parity of the small-layer path (hidden <= 1024 and a few thousand neurons,
one or two tokens per pass: one thread-block cluster per call) against the
oracle, through the C ABI.

Cases: one and two tokens per pass and each register layout (H <= 256, 512,
1024), bf16 and fp32 activations, a hidden size that is not a multiple of the
warp's vector stride, intermediate sizes that leave CTAs of the cluster partly
filled or empty, the largest layer the path takes at H = 1024 and one just
beyond it (the persistent kernel), thresholds 0 and +inf, calls without index
lists, repeated calls, and one workspace shared with the persistent decode
kernel of a wider layer between two small calls.
"""
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


def _t(oracle, w, H, k):
    if k is None:
        return 0.0
    if k == "inf":
        return float("inf")
    cal = oracle.bf16_to_f64(inputs.activations_bf16(8, H, seed=inputs.SEED_CALIB))
    return float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), k)))


def _call(sats, layer, ws, x, t, B, H, N, f32, lists=True):
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda") if lists else None
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda") if lists else None
    (sats.sparse_mlp_f32 if f32 else sats.sparse_mlp)(layer, x, t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    return y, idx, cnt


@pytest.mark.parametrize("H,N,B,k,f32", [
    (512, 1408, 1, 0.5, False),     # the small-layer workload's shape
    (512, 1408, 2, 0.7, False),     # two tokens in one pass
    (512, 1408, 2, 0.5, True),      # fp32 activations
    (128, 300, 1, 0.6, False),      # one vector per lane; 300 = 9 CTAs of 32 + 12
    (264, 95, 2, 0.5, True),        # H not a multiple of 256 (lanes 1..31 idle on the second vector)
    (1024, 1536, 2, 0.9, False),    # four vectors per lane; the largest layer of the path at H = 1024
    (1024, 1600, 1, 0.5, False),    # just beyond it: the persistent kernel
    (1024, 777, 1, 0.3, True),
    (64, 5, 2, 0.5, False),         # five neurons: most CTAs of the cluster own none
])
def test_small_layer_matches_oracle(sats, oracle, H, N, B, k, f32):
    assert sats.uses_tensor_cores(H, B) == 0
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + H + N)
    t = _t(oracle, w, H, k)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    if f32:
        xh = inputs.activations_f32(B, H, seed=inputs.SEED_X + 3)
        x64, x = xh.astype(np.float64), P.dev(xh)
    else:
        xh = inputs.activations_bf16(B, H, seed=inputs.SEED_X + 3)
        x64, x = oracle.bf16_to_f64(xh), P.dev_u16(xh)
    for rep in range(3):        # repeated calls on one workspace
        y, idx, cnt = _call(sats, layer, ws, x, t, B, H, N, f32)
        keep = P.keep_from_lists(idx, cnt, N)
        y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t, keep_hint=keep,
                                                     band_rel=P.BAND_REL)
        P.assert_keep_match(keep, keep_ref, a_ref, t)
        P.assert_close(y.cpu().numpy(), y_ref)
    y2, _, _ = _call(sats, layer, ws, x, t, B, H, N, f32, lists=False)
    P.assert_close(y2.cpu().numpy(), y_ref)
    layer.close()


@pytest.mark.parametrize("k", [None, "inf"])
def test_small_layer_threshold_zero_and_inf(sats, oracle, k):
    H, N, B = 512, 1408, 2
    w = inputs.mlp_weights(H, N)
    xh = inputs.activations_bf16(B, H)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    y, idx, cnt = _call(sats, layer, ws, P.dev_u16(xh), _t(oracle, w, H, k), B, H, N, False)
    keep = P.keep_from_lists(idx, cnt, N)
    if k is None:
        assert keep.all()
        P.assert_close(y.cpu().numpy(), oracle.dense_mlp(oracle.bf16_to_f64(xh), w.Wg, w.Wu, w.Wd))
    else:
        assert not keep.any() and np.all(y.cpu().numpy() == 0.0)
    layer.close()


def test_small_and_persistent_kernels_share_a_workspace(sats, oracle):
    # a small layer, then a wide one (the persistent decode kernel), then the small one again,
    # on one workspace large enough for both
    shapes = [(512, 1408), (2048, 700)]
    ws = sats.Workspace(2048, 1408, 1)
    layers, ws_w, ts, xs = [], [], [], []
    for H, N in shapes:
        w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + 5 * H)
        layers.append(sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd)))
        ws_w.append(w)
        ts.append(_t(oracle, w, H, 0.6))
        xs.append(inputs.activations_bf16(1, H, seed=inputs.SEED_X + H))
    for i in (0, 1, 0, 1):
        H, N = shapes[i]
        w = ws_w[i]
        y, idx, cnt = _call(sats, layers[i], ws, P.dev_u16(xs[i]), ts[i], 1, H, N, False)
        keep = P.keep_from_lists(idx, cnt, N)
        y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xs[i]), w.Wg, w.Wu, w.Wd, ts[i],
                                                     keep_hint=keep, band_rel=P.BAND_REL)
        P.assert_keep_match(keep, keep_ref, a_ref, ts[i])
        P.assert_close(y.cpu().numpy(), y_ref)
    for l in layers:
        l.close()
