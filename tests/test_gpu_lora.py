"""GPU parity of the LoRA-aware sparse path (sats_sparse_mlp_lora; Sec. 4, the
sparse path of a fine-tuned model on its adapted weights W + s A B) against the
oracle's factor-by-factor statement, element by element, plus the kept lists."""
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


def _threshold(oracle, w, H, k):
    cal = oracle.bf16_to_f64(inputs.activations_bf16(8, H, seed=inputs.SEED_CALIB))
    return float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), k)))


def _setup(sats, H, N, r, scale, seed=0):
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + seed)
    lo = inputs.lora_adapter(H, N, r, seed=7000 + seed)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    lora = sats.Lora(layer, *(P.dev_u16(m) for m in lo), scale=scale)
    return w, lo, layer, lora


def _call(sats, layer, lora, xdev, t, B, H, N, ws):
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    sats.sparse_mlp_lora(layer, lora, xdev, t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    return y.cpu().numpy(), P.keep_from_lists(idx, cnt, N)


@pytest.mark.parametrize("H,N,B,r,k,f32", [
    (512, 1408, 1, 16, 0.5, False),
    (4096, 2048, 2, 32, 0.7, False),    # two tokens in one pass, the largest rank
    (1024, 777, 1, 8, 0.9, False),      # ragged chunk tail, the smallest rank
    (8192, 300, 1, 24, 0.5, False),     # four vectors per thread; 24 = a rank not a power of two
    (2048, 1000, 2, 16, 0.6, True),     # fp32 x
    (512, 1408, 5, 16, 0.5, False),     # three passes of the decode kernel
])
def test_lora_matches_oracle(sats, oracle, H, N, B, r, k, f32):
    scale = 0.5
    w, lo, layer, lora = _setup(sats, H, N, r, scale)
    t = _threshold(oracle, w, H, k)
    ws = sats.Workspace(H, N, B)
    if f32:
        xf = inputs.activations_f32(B, H, seed=inputs.SEED_X + 1)
        x64, xdev = xf.astype(np.float64), P.dev(xf)
    else:
        xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + 1)
        x64, xdev = oracle.bf16_to_f64(xb), P.dev_u16(xb)
    y, keep = _call(sats, layer, lora, xdev, t, B, H, N, ws)
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp_lora(x64, w.Wg, w.Wu, w.Wd, lo, scale, t, keep_hint=keep,
                                                      band_rel=P.BAND_REL)
    P.assert_keep_match(keep, keep_ref, a_ref, t)
    P.assert_close(y, y_ref)
    # the adapter changes the result (this is not the base MLP)
    y_base, *_ = oracle.sparse_mlp(x64, w.Wg, w.Wu, w.Wd, t)
    assert np.linalg.norm(y_ref - y_base) > 1e-3 * np.linalg.norm(y_base)
    lora.close()
    layer.close()


def test_lora_scale_zero_is_the_base_path(sats, oracle):
    H, N, B = 1024, 2000, 2
    w, lo, layer, lora = _setup(sats, H, N, 16, 0.0, seed=3)
    t = _threshold(oracle, w, H, 0.7)
    xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + 5)
    ws = sats.Workspace(H, N, B)
    y, keep = _call(sats, layer, lora, P.dev_u16(xb), t, B, H, N, ws)
    y0 = torch.empty(B, H, dtype=torch.float32, device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    sats.sparse_mlp(layer, P.dev_u16(xb), t, y0, ws, idx, cnt)
    assert np.array_equal(keep, P.keep_from_lists(idx, cnt, N))
    np.testing.assert_allclose(y, y0.cpu().numpy(), rtol=1e-5, atol=1e-6)
    lora.close()
    layer.close()


def test_lora_repeat_and_interleave(sats, oracle):
    """The x A sums are cleared after every call: repeated LoRA calls, and base
    calls in between on the same workspace, give the same LoRA result."""
    H, N, B = 2048, 1500, 1
    w, lo, layer, lora = _setup(sats, H, N, 16, 1.0, seed=4)
    t = _threshold(oracle, w, H, 0.5)
    xb = inputs.activations_bf16(B, H, seed=inputs.SEED_X + 6)
    ws = sats.Workspace(H, N, B)
    y1, k1 = _call(sats, layer, lora, P.dev_u16(xb), t, B, H, N, ws)
    ybase = torch.empty(B, H, dtype=torch.float32, device="cuda")
    for _ in range(3):
        y2, k2 = _call(sats, layer, lora, P.dev_u16(xb), t, B, H, N, ws)
        sats.sparse_mlp(layer, P.dev_u16(xb), t, ybase, ws)
        assert np.array_equal(k1, k2)
        np.testing.assert_allclose(y2, y1, rtol=1e-5, atol=1e-6)
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp_lora(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, lo, 1.0, t,
                                                      keep_hint=k1, band_rel=P.BAND_REL)
    P.assert_close(y1, y_ref)
    lora.close()
    layer.close()


def test_lora_llama_layer(sats, oracle):
    """Hidden 4096 / intermediate 14336, rank 16, one decode token at 50 / 90 %."""
    H, N, r = inputs.LLAMA_H, inputs.LLAMA_N, 16
    w, lo, layer, lora = _setup(sats, H, N, r, 1.0, seed=5)
    ws = sats.Workspace(H, N, 1)
    xb = inputs.activations_bf16(1, H, seed=inputs.SEED_X + 7)
    for k in (0.5, 0.9):
        t = _threshold(oracle, w, H, k)
        y, keep = _call(sats, layer, lora, P.dev_u16(xb), t, 1, H, N, ws)
        y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp_lora(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, lo, 1.0, t,
                                                          keep_hint=keep, band_rel=P.BAND_REL)
        P.assert_keep_match(keep, keep_ref, a_ref, t)
        P.assert_close(y, y_ref)
    lora.close()
    layer.close()


def test_lora_argument_errors(sats):
    H, N = 64, 64
    z = torch.zeros(H, N, dtype=torch.int16, device="cuda")
    layer = sats.Layer(z, z, torch.zeros(N, H, dtype=torch.int16, device="cuda"))
    for r in (4, 12, 40):
        a = torch.zeros(H, r, dtype=torch.int16, device="cuda")
        b = torch.zeros(r, N, dtype=torch.int16, device="cuda")
        with pytest.raises(sats.SatsError) as e:
            sats.Lora(layer, a, b, a, b, torch.zeros(N, r, dtype=torch.int16, device="cuda"),
                      torch.zeros(r, H, dtype=torch.int16, device="cuda"))
        assert e.value.status == sats.ESHAPE
    layer.close()
