"""Failure detection without a GPU fault: the library's bounded device waits,
run on conditions nothing satisfies (an mbarrier phase no thread completes, a
workspace counter no CTA raises), give up after their time limit and report
SATS_ETIMEOUT through the workspace status word; the status is read and
cleared, and the same workspace then serves a normal call, checked against the
oracle (Sec. 2, Eqs. 1-5)."""
import time

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


def test_bounded_waits_time_out_and_the_workspace_recovers(sats, oracle):
    H, N = 512, 1408
    w = inputs.mlp_weights(H, N, seed=inputs.SEED_WEIGHTS + 9)
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    ws = sats.Workspace(H, N, 1)
    assert sats.get_error(ws) == sats.OK
    t0 = time.perf_counter()
    sats.selftest_wait_timeout(ws)
    status = sats.get_error(ws)
    elapsed = time.perf_counter() - t0
    assert status == sats.ETIMEOUT
    assert elapsed >= 3.5          # both waits ran to their 2 s limit
    assert sats.get_error(ws) == sats.OK   # read and cleared
    # the workspace and the device stay usable
    cal = oracle.bf16_to_f64(inputs.activations_bf16(8, H, seed=inputs.SEED_CALIB))
    t = float(np.float32(oracle.percentile_threshold(oracle.gate_act(cal, w.Wg), 0.5)))
    xb = inputs.activations_bf16(1, H, seed=inputs.SEED_X + 9)
    y = torch.full((1, H), float("nan"), dtype=torch.float32, device="cuda")
    idx = torch.full((1, N), -1, dtype=torch.int32, device="cuda")
    cnt = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    sats.sparse_mlp(layer, P.dev_u16(xb), t, y, ws, idx, cnt)
    assert sats.get_error(ws) == sats.OK
    keep = P.keep_from_lists(idx, cnt, N)
    y_ref, a_ref, keep_ref, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, t, keep_hint=keep,
                                                 band_rel=P.BAND_REL)
    P.assert_keep_match(keep, keep_ref, a_ref, t)
    P.assert_close(y.cpu().numpy(), y_ref)
    layer.close()
