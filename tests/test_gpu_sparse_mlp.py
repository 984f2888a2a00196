"""GPU parity of the thresholded gated MLP (Sec. 2, Eqs. 1-5) against the oracle.

Every case runs the CUDA path through the C ABI on seeded inputs and compares
element by element with the fp64 oracle on the same bf16 values (rules in
tests/_parity.py).
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


def _threshold(oracle, w, H, k, n_cal=8, seed=inputs.SEED_CALIB):
    if k is None:
        return 0.0
    if k == "inf":
        return float("inf")
    cal = oracle.bf16_to_f64(inputs.activations_bf16(n_cal, H, seed=seed))
    return float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), k)))


def _run(sats, oracle, H, N, B, k, seed=0, f32=False, want_lists=True):
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + 17 * seed)
    t = _threshold(oracle, w, H, k)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, max(B, 1))
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda") if want_lists else None
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda") if want_lists else None
    if f32:
        xf = inputs.activations_f32(B, H, seed=inputs.SEED_X + seed)
        x64 = xf.astype(np.float64)
        sats.sparse_mlp_f32(layer, P.dev(xf), t, y, ws, idx, cnt)
    else:
        xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + seed)
        x64 = oracle.bf16_to_f64(xb)
        sats.sparse_mlp(layer, P.dev_u16(xb), t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    y_gpu = y.cpu().numpy()
    if want_lists:
        keep_gpu = P.keep_from_lists(idx, cnt, N)
        y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t, keep_hint=keep_gpu,
                                                     band_rel=P.BAND_REL)
        P.assert_keep_match(keep_gpu, keep_ref, a_ref, t)
    else:
        y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t)
    P.assert_close(y_gpu, y_ref)
    layer.close()
    return keep_ref, y_gpu


@pytest.mark.parametrize("H,N,B,k", [
    (512, 1408, 1, 0.5),        # hidden 512 / intermediate 1408 layer, one token
    (64, 100, 1, 0.5),          # ragged chunk tail (100 = 6 * 16 + 4)
    (8, 1, 1, 0.5),             # one neuron, one vector per row
    (8, 17, 3, 0.3),            # three tokens in one pass
    (256, 333, 2, 0.7),
    (512, 1408, 4, 0.5),        # four tokens: one full pass
    (512, 1408, 5, 0.5),        # five tokens: two passes
    (520, 200, 9, 0.6),         # H not a multiple of the thread count; three passes
    (2048, 700, 1, 0.9),
    (2560, 1003, 2, 0.6),       # three gate rows per 16 KB stage (chunks of 3 + 3 + 2 rows; a 3-row tail)
    (4096, 640, 4, 0.5),        # two vectors per consumer thread
    (6144, 300, 3, 0.5),        # four vectors per consumer thread, passes of two
    (8192, 130, 2, 0.5),        # the largest hidden size
    (64, 100003, 1, 0.7),       # slices of more than 64 chunks (index words re-read, not kept in shared memory)
    (64, 100003, 2, 0.5),
])
def test_sparse_mlp_matches_oracle(sats, oracle, H, N, B, k):
    keep, _ = _run(sats, oracle, H, N, B, k)
    if k is not None and N > 50:
        frac = 1.0 - keep.mean()
        assert 0.05 < frac < 0.98


@pytest.mark.parametrize("B", [2, 5])
def test_threshold_zero_keeps_all_and_inf_keeps_none(sats, oracle, B):
    keep, _ = _run(sats, oracle, 512, 1408, B, None)
    assert keep.all()
    keep, y = _run(sats, oracle, 512, 1408, B, "inf")
    assert not keep.any() and np.all(y == 0.0)


@pytest.mark.parametrize("H,N,B,k", [
    (136, 77, 5, 0.5),          # K = 136 (a partial 64-wide K block), N = 77 (h rows padded to 80)
    (512, 1408, 8, 0.5),
    (512, 1408, 129, 0.7),      # two 128-token tiles, the second with one token
    (1024, 2000, 300, 0.9),     # 2000 = 20 full 96-neuron tiles + 80
    (4096, 640, 3, 0.5),        # the smallest batch that leaves the fused kernel at H = 4096
])
def test_tensor_core_batches_match_oracle(sats, oracle, H, N, B, k):
    assert sats.uses_tensor_cores(H, B)
    keep, _ = _run(sats, oracle, H, N, B, k)
    frac = 1.0 - keep.mean()
    assert abs(frac - k) < 0.1


@pytest.mark.parametrize("H,N,B", [
    (4096, 640, 3),     # 16 token columns: hi and lo parts in one MMA of N = 32
    (1024, 777, 40),
    (512, 1408, 128),   # 128 columns: the largest merged MMA (N = 256; 512 TMEM columns)
    (512, 1408, 200),   # 208 columns: two MMAs per step, hi and lo into the same accumulator
    (1024, 777, 240),   # above 224 fp32 tokens: the prefill kernels, the second token tile partial
])
def test_tensor_core_fp32_activations(sats, oracle, H, N, B):
    """fp32 x split into bf16 hi + lo parts: the gate keeps ~fp32 accuracy."""
    assert sats.uses_tensor_cores(H, B)
    _run(sats, oracle, H, N, B, 0.5, f32=True)


@pytest.mark.parametrize("B,k", [(8, 0.5), (64, 0.7), (256, 0.9), (2048, 0.5)])
def test_llama_layer_batches_sampled(sats, oracle, B, k):
    """Hidden 4096 / intermediate 14336 at decode and prefill batch sizes: every
    token's kept count is checked against its list, and a sample of tokens
    (first, last and four seeded others) element by element against the oracle."""
    H, N = inputs.LLAMA_H, inputs.LLAMA_N
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + 5)
    t = _threshold(oracle, w, H, k)
    xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + B)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    sats.sparse_mlp(layer, P.dev_u16(xb), t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    layer.close()
    rng = np.random.default_rng(B)
    rows = sorted(set([0, B - 1] + rng.choice(B, size=min(B, 4), replace=False).tolist()))
    keep_gpu = P.keep_from_lists(idx[rows], cnt[rows], N)
    x64 = oracle.bf16_to_f64(xb[rows])
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t, keep_hint=keep_gpu,
                                                 band_rel=P.BAND_REL)
    P.assert_keep_match(keep_gpu, keep_ref, a_ref, t)
    P.assert_close(y[rows].cpu().numpy(), y_ref)
    c = cnt.cpu().numpy()
    assert np.all((c >= 0) & (c <= N))
    assert abs((1.0 - c.mean() / N) - k) < 0.05


def test_fp32_activations(sats, oracle):
    _run(sats, oracle, 1024, 777, 3, 0.5, f32=True)


def test_without_index_lists(sats, oracle):
    _run(sats, oracle, 512, 1408, 3, 0.5, want_lists=False)


def test_dense_mlp_matches_oracle(sats, oracle):
    H, N, B = 512, 1408, 3
    w = inputs.mlp_weights(H, N)
    xb = inputs.activations_bf16(B, H)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    y = torch.empty(B, H, dtype=torch.float32, device="cuda")
    sats.dense_mlp(layer, P.dev_u16(xb), y, ws)
    assert sats.get_error(ws) == sats.OK
    P.assert_close(y.cpu().numpy(), oracle.dense_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd))


def test_skipped_rows_are_not_read(sats, oracle):
    """Poisoning W_up columns / W_down rows of neurons no token keeps leaves y unchanged."""
    H, N, B = 512, 1408, 2
    w = inputs.mlp_weights(H, N)
    xb = inputs.activations_bf16(B, H)
    t = _threshold(oracle, w, H, 0.7)
    _, a_ref, keep, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, t)
    near = P.band_mask(a_ref, t).any(axis=0)
    off = np.where((keep.max(axis=0) == 0) & ~near)[0]
    assert off.size > 100
    Wu2, Wd2 = w.Wu.copy(), w.Wd.copy()
    Wu2[:, off] = 0x7FC0          # bf16 NaN
    Wd2[off, :] = 0x7FC0
    ys = []
    for Wu, Wd in ((w.Wu, w.Wd), (Wu2, Wd2)):
        layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(Wu), P.dev_u16(Wd))
        ws = sats.Workspace(H, N, B)
        y = torch.empty(B, H, dtype=torch.float32, device="cuda")
        sats.sparse_mlp(layer, P.dev_u16(xb), t, y, ws)
        ys.append(y.cpu().numpy())
        layer.close()
    # chunks are claimed dynamically, so the fp32 grouping of the sum over kept
    # neurons (and its last bits) may differ between calls; nothing else may
    assert np.all(np.isfinite(ys[1]))
    np.testing.assert_allclose(ys[1], ys[0], rtol=1e-5, atol=1e-6)


def test_repeat_calls_agree(sats):
    H, N, B = 512, 1408, 3
    w = inputs.mlp_weights(H, N)
    xb = P.dev_u16(inputs.activations_bf16(B, H))
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    outs, lists = [], []
    for _ in range(3):
        y = torch.empty(B, H, dtype=torch.float32, device="cuda")
        idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        sats.sparse_mlp(layer, xb, 0.2, y, ws, idx, cnt)
        outs.append(y.cpu().numpy())
        lists.append(P.keep_from_lists(idx, cnt, N))
    for i in (1, 2):
        assert np.array_equal(lists[0], lists[i])          # the kept sets are exactly reproducible
        np.testing.assert_allclose(outs[i], outs[0], rtol=1e-5, atol=1e-6)


def test_argument_errors(sats):
    H, N = 64, 4096
    w = inputs.mlp_weights(H, N)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, 1)
    x = P.dev_u16(inputs.activations_bf16(1, H))
    y = torch.empty(1, H, dtype=torch.float32, device="cuda")
    for bad_t in (float("nan"), -0.5):
        with pytest.raises(sats.SatsError) as e:
            sats.sparse_mlp(layer, x, bad_t, y, ws)
        assert e.value.status == sats.EINVAL
    small = sats.Workspace(8, 8, 1)
    with pytest.raises(sats.SatsError) as e:
        sats.sparse_mlp(layer, x, 0.1, y, small)
    assert e.value.status == sats.ENOSPACE
    with pytest.raises(sats.SatsError):
        sats.Layer(P.dev_u16(np.zeros((12, 8), np.uint16)), P.dev_u16(np.zeros((12, 8), np.uint16)),
                   P.dev_u16(np.zeros((8, 12), np.uint16)))
    # B = 0 is a no-op
    sats.sparse_mlp(layer, x[:0], 0.1, y[:0], ws)
    assert sats.get_error(ws) == sats.OK


@pytest.mark.parametrize("k", [0.5, 0.7, 0.9])
def test_llama_layer_full_size(sats, oracle, k):
    """Hidden 4096 / intermediate 14336, one decode token, the bench's launch."""
    keep, _ = _run(sats, oracle, inputs.LLAMA_H, inputs.LLAMA_N, 1, k, seed=3)
    assert abs((1.0 - keep.mean()) - k) < 0.05
