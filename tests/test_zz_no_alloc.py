"""The workspace-free entry point, sats_sparse_mlp_fixed_scratch.

It serves callers that cannot allocate device memory (for example a plug-in
whose host application owns every allocation, or a plain C caller with no
device allocator): instead of a caller workspace it uses a 256 KiB array in
the library's own device memory.  These tests call it through the C ABI and
check that two calls in a row give what the workspace entry point gives on the
same inputs, that both agree with the CPU oracle (kept sets outside the
threshold band, y within the tolerance), that the call reports its device
status through the caller's status word, and that a shape needing more
scratch than the array holds is refused.  The file is named so that pytest
collects it last.
"""
import numpy as np
import pytest
import torch

from paper_2607_08991_gb300 import inputs
from tests import _parity as P

pytestmark = pytest.mark.gpu

FIXED_SCRATCH_BYTES = 1 << 18


@pytest.fixture(scope="module")
def sats():
    import __graft_entry__
    __graft_entry__.build()
    from paper_2607_08991_gb300 import sats as s
    return s


@pytest.mark.parametrize("H,N,B,k", [(512, 1408, 1, 0.5), (4096, 14336, 1, 0.7), (1024, 777, 3, 0.5)])
def test_fixed_scratch_matches_workspace_entry(sats, oracle, H, N, B, k):
    w = inputs.mlp_weights(H, N)
    xb = inputs.activations_bf16(B, H)
    cal = oracle.bf16_to_f64(inputs.activations_bf16(8, H, seed=inputs.SEED_CALIB))
    t = float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), k)))
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    x = P.dev_u16(xb)

    ws = sats.Workspace(H, N, B)
    y_ref = torch.empty(B, H, dtype=torch.float32, device="cuda")
    idx_ref = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt_ref = torch.empty(B, dtype=torch.int32, device="cuda")
    sats.sparse_mlp(layer, x, t, y_ref, ws, idx_ref, cnt_ref)
    assert sats.get_error(ws) == sats.OK
    keep_ref = P.keep_from_lists(idx_ref, cnt_ref, N)

    # the oracle on the same inputs, taking the kernel's decisions inside the threshold band only
    y_or, a_or, keep_or, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, t,
                                               keep_hint=keep_ref, band_rel=P.BAND_REL)
    P.assert_keep_match(keep_ref, keep_or, a_or, t)

    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    for _ in range(2):          # two calls in a row share the library's scratch
        y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
        idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        sats.sparse_mlp_fixed_scratch(layer, x, t, y, idx, cnt, dev_status=status)
        torch.cuda.synchronize()
        assert sats.get_status_word(status) == sats.OK
        keep = P.keep_from_lists(idx, cnt, N)
        assert np.array_equal(keep, keep_ref)
        P.assert_close(y.cpu().numpy(), y_ref.cpu().numpy())
        P.assert_close(y.cpu().numpy(), y_or)
    layer.close()


def test_fixed_scratch_refuses_shapes_beyond_its_limit(sats):
    H, N = 8, 300000            # one 64-bit index word per 8 neurons: about 300 KB > 256 KiB
    z = torch.zeros(H, N, dtype=torch.int16, device="cuda")
    layer = sats.Layer(z, z, torch.zeros(N, H, dtype=torch.int16, device="cuda"))
    x = torch.zeros(1, H, dtype=torch.int16, device="cuda")
    y = torch.empty(1, H, dtype=torch.float32, device="cuda")
    with pytest.raises(sats.SatsError) as e:
        sats.sparse_mlp_fixed_scratch(layer, x, 0.5, y)
    assert e.value.status == sats.ENOSPACE
    layer.close()


def test_fixed_scratch_two_tokens_of_a_wide_layer(sats, oracle):
    # H = 8192 runs one token per pass of the fused kernel, so B = 2 takes the tensor-core path and
    # needs its staging; the call either fits in the array and matches the workspace entry, or is
    # refused with SATS_ENOSPACE, as sats_workspace_bytes says
    H, N, B = 8192, 64, 2
    w = inputs.mlp_weights(H, N)
    xb = inputs.activations_bf16(B, H)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    x = P.dev_u16(xb)
    y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
    need = int(sats.lib().sats_workspace_bytes(H, N, B))
    assert sats.uses_tensor_cores(H, B) and need > 0
    if need > FIXED_SCRATCH_BYTES:
        with pytest.raises(sats.SatsError) as e:
            sats.sparse_mlp_fixed_scratch(layer, x, 0.0, y)
        assert e.value.status == sats.ENOSPACE
    else:
        status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        sats.sparse_mlp_fixed_scratch(layer, x, 0.0, y, dev_status=status)
        assert sats.get_status_word(status) == sats.OK
        y_or = oracle.dense_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd)
        P.assert_close(y.cpu().numpy(), y_or)
    layer.close()
