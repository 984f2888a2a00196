"""GPU parity of the union path (sats_sparse_mlp_union) for batches of 3 to 8
tokens with one threshold and hidden size up to 4096: the gate on the tensor
cores, then the up and down projections only for the union of the tokens' kept
neurons (Sec. 2, Eqs. 1-5 per token; the union is a scheduling choice, not a
change of the result).  Each case is compared element by element with the fp64
oracle; poisoned rows outside the union show that they are not read.
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


def _threshold(oracle, w, H, k, n_cal=8):
    cal = oracle.bf16_to_f64(inputs.activations_bf16(n_cal, H, seed=inputs.SEED_CALIB))
    return float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), k)))


def _case(sats, oracle, H, N, B, k, f32=False, seed=3, wmod=None):
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + seed)
    t = _threshold(oracle, w, H, k) if k != "inf" else float("inf")
    Wu, Wd = (w.Wu, w.Wd) if wmod is None else wmod(w)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(Wu), P.dev_u16(Wd))
    ws = sats.Workspace(H, N, B)
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    if f32:
        xf = inputs.activations_f32(B, H, seed=inputs.SEED_X + seed)
        x64 = xf.astype(np.float64)
        sats.sparse_mlp_union(layer, P.dev(xf), t, y, ws, idx, cnt)
    else:
        xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + seed)
        x64 = oracle.bf16_to_f64(xb)
        sats.sparse_mlp_union(layer, P.dev_u16(xb), t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    layer.close()
    keep_gpu = P.keep_from_lists(idx, cnt, N)
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t, keep_hint=keep_gpu, band_rel=P.BAND_REL)
    P.assert_keep_match(keep_gpu, keep_ref, a_ref, t)
    return y.cpu().numpy(), y_ref, keep_gpu, a_ref, t


@pytest.mark.parametrize("H,N,B,k,f32", [
    (512, 1408, 3, 0.9, False),      # the smallest union batch at H = 512
    (4096, 2048, 8, 0.9, False),     # the largest union batch at the largest union hidden size
    (1024, 3000, 7, 0.95, True),     # fp32 x (bf16 hi + lo)
    (2048, 1000, 4, 0.8, False),
    (136, 77, 6, 0.5, False),        # 17 of 512 threads cover the hidden units; a partial last stage
    (4096, 5000, 5, 0.7, True),
])
def test_union_batches_match_oracle(sats, oracle, H, N, B, k, f32):
    assert sats.uses_tensor_cores(H, B)
    y, y_ref, keep, _, _ = _case(sats, oracle, H, N, B, k, f32=f32)
    P.assert_close(y, y_ref)
    union = keep.any(axis=0).mean()
    assert 0.0 < union < 1.0 or N < 100


def test_union_shape_limits(sats):
    """Outside 3 <= B <= 8 or above H = 4096 the union entry refuses the call."""
    for H, B in ((512, 2), (512, 9), (8192, 4)):
        N = 64
        z = torch.zeros(H, N, dtype=torch.int16, device="cuda")
        layer = sats.Layer(z, z, torch.zeros(N, H, dtype=torch.int16, device="cuda"))
        ws = sats.Workspace(H, N, max(B, 3))
        x = torch.zeros(B, H, dtype=torch.int16, device="cuda")
        y = torch.empty(B, H, dtype=torch.float32, device="cuda")
        with pytest.raises(sats.SatsError) as e:
            sats.sparse_mlp_union(layer, x, 0.5, y, ws)
        assert e.value.status == sats.ESHAPE
        layer.close()


def test_union_rows_outside_are_not_read(sats, oracle):
    """NaN in the W_up columns and W_down rows of every neuron outside the union
    (away from the threshold band) leaves y finite and unchanged."""
    H, N, B, k = 1024, 4096, 8, 0.95
    y0, _, keep, a_ref, t = _case(sats, oracle, H, N, B, k)
    near = P.band_mask(a_ref, t).any(axis=0)
    off = np.where(~keep.any(axis=0) & ~near)[0]
    assert off.size > N // 4

    def poison(w):
        Wu2, Wd2 = w.Wu.copy(), w.Wd.copy()
        Wu2[:, off] = 0x7FC0   # bf16 NaN
        Wd2[off, :] = 0x7FC0
        return Wu2, Wd2

    y1, _, _, _, _ = _case(sats, oracle, H, N, B, k, wmod=poison)
    assert np.all(np.isfinite(y1))
    # the CTAs add their y partials in L2 in any order, so the last bits may differ between calls
    np.testing.assert_allclose(y1, y0, rtol=1e-5, atol=1e-6)


def test_union_empty(sats, oracle):
    """t = inf keeps nothing: the union is empty, y is zero and every list is empty."""
    y, y_ref, keep, _, _ = _case(sats, oracle, 512, 1408, 6, "inf")
    assert not keep.any()
    assert np.all(y == 0.0) and np.all(y_ref == 0.0)


def test_union_llama_layer_sampled(sats, oracle):
    """Hidden 4096 / intermediate 14336, 8 tokens at 90 %: kept counts for every
    token, and three tokens element by element."""
    H, N, B, k = inputs.LLAMA_H, inputs.LLAMA_N, 8, 0.9
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + 5)
    t = _threshold(oracle, w, H, k)
    xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + 77)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    sats.sparse_mlp_union(layer, P.dev_u16(xb), t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    layer.close()
    rows = [0, 5, B - 1]
    keep_gpu = P.keep_from_lists(idx[rows], cnt[rows], N)
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb[rows]), w.Wg, w.Wu, w.Wd, t,
                                                 keep_hint=keep_gpu, band_rel=P.BAND_REL)
    P.assert_keep_match(keep_gpu, keep_ref, a_ref, t)
    P.assert_close(y[rows].cpu().numpy(), y_ref)
    c = cnt.cpu().numpy()
    assert abs((1.0 - c.mean() / N) - k) < 0.05
