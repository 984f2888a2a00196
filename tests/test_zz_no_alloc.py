"""The workspace-free entry point, sats_sparse_mlp_fixed_scratch.

It serves callers that cannot allocate device memory (for example a plug-in
whose host application owns every allocation, or a plain C caller with no
device allocator): instead of a caller workspace it uses a 1 MiB array in the
library's own device memory.  These tests call it through the C ABI and check
that two calls in a row give what the workspace entry point gives on the same
inputs, and that a shape needing more scratch than the array holds is refused.
The file is named so that pytest collects it last.
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

    for _ in range(2):          # two calls in a row share the library's scratch
        y = torch.full((B, H), float("nan"), dtype=torch.float32, device="cuda")
        idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
        cnt = torch.empty(B, dtype=torch.int32, device="cuda")
        sats.sparse_mlp_fixed_scratch(layer, x, t, y, idx, cnt)
        torch.cuda.synchronize()
        assert np.array_equal(P.keep_from_lists(idx, cnt, N), keep_ref)
        P.assert_close(y.cpu().numpy(), y_ref.cpu().numpy())
    layer.close()


def test_fixed_scratch_refuses_shapes_beyond_its_limit(sats):
    H, N = 8, 300000            # one flag byte per neuron: 300 KB > 256 KiB
    z = torch.zeros(H, N, dtype=torch.int16, device="cuda")
    layer = sats.Layer(z, z, torch.zeros(N, H, dtype=torch.int16, device="cuda"))
    x = torch.zeros(1, H, dtype=torch.int16, device="cuda")
    y = torch.empty(1, H, dtype=torch.float32, device="cuda")
    with pytest.raises(sats.SatsError) as e:
        sats.sparse_mlp_fixed_scratch(layer, x, 0.5, y)
    assert e.value.status == sats.ENOSPACE
    layer.close()
