"""Calls captured into a CUDA graph and replayed give what the same calls give
when issued directly: the library records only stream work (kernels, and a
memset on the tensor-core prefill path), so a serving loop can capture a
decode step once and replay it."""
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


@pytest.mark.parametrize("H,N,B", [(512, 1408, 1), (512, 1408, 2), (1024, 2000, 40), (512, 1408, 300)])
def test_sparse_mlp_replays_in_a_graph(sats, H, N, B):
    w = inputs.mlp_weights(H, N)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, B)
    x = P.dev_u16(inputs.activations_bf16(B, H))
    y_ref = torch.empty(B, H, device="cuda")
    idx_ref = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt_ref = torch.empty(B, dtype=torch.int32, device="cuda")
    sats.sparse_mlp(layer, x, 0.2, y_ref, ws, idx_ref, cnt_ref)
    torch.cuda.synchronize()

    y = torch.full((B, H), float("nan"), device="cuda")
    idx = torch.full((B, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((B,), -1, dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        sats.sparse_mlp(layer, x, 0.2, y, ws, idx, cnt, stream=s)
    torch.cuda.synchronize()
    assert torch.isnan(y).all()          # capture records work; it runs nothing
    for _ in range(3):
        y.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert sats.get_error(ws) == sats.OK
        assert np.array_equal(P.keep_from_lists(idx, cnt, N), P.keep_from_lists(idx_ref, cnt_ref, N))
        np.testing.assert_allclose(y.cpu().numpy(), y_ref.cpu().numpy(), rtol=1e-5, atol=1e-6)
    layer.close()


def test_routed_stack_replays_in_a_graph(sats):
    L, H, N, B, V = 3, 512, 1408, 8, 1000
    ws_ = [inputs.mlp_weights(H, N, layer=l) for l in range(L)]
    layers = [sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd)) for w in ws_]
    nw = [P.dev(inputs.norm_weight(H, layer=l)) for l in range(L)]
    lut = P.dev(inputs.routing_lut(V, 0.3))
    ids = P.dev(inputs.token_ids_uniform(B, V))
    x0 = P.dev(inputs.activations_f32(B, H))
    ws = sats.Workspace(H, N, B)
    x_ref = x0.clone()
    sats.mlp_stack(layers, nw, [0.2, 0.25, 0.3], 1e-5, x_ref, ws, token_ids=ids, lut=lut)
    torch.cuda.synchronize()

    x = x0.clone()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        sats.mlp_stack(layers, nw, [0.2, 0.25, 0.3], 1e-5, x, ws, token_ids=ids, lut=lut, stream=s)
    for _ in range(2):
        x.copy_(x0)
        g.replay()
        torch.cuda.synchronize()
        assert sats.get_error(ws) == sats.OK
        np.testing.assert_allclose(x.cpu().numpy(), x_ref.cpu().numpy(), rtol=1e-5, atol=1e-5)
    for l in layers:
        l.close()
