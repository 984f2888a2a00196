"""The C-ABI library builds, loads and exports every symbol include/sats.h
declares; host-side argument checks answer without touching a GPU."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libsats():
    from paper_2607_08991_gb300 import build
    path = build.build_library()
    return ctypes.CDLL(path)


def _declared():
    src = open(os.path.join(ROOT, "include", "sats.h")).read()
    return sorted(set(re.findall(r"SATS_API[^;(]*?\b(sats_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for required in ("sats_sparse_mlp", "sats_route", "sats_mlp_stack", "sats_dense_mlp", "sats_layer_create"):
        assert required in names


def test_every_declared_symbol_is_exported(libsats):
    for name in _declared():
        assert hasattr(libsats, name), name


def test_binding_covers_every_symbol():
    from paper_2607_08991_gb300 import sats
    assert sorted(sats.exported_symbols()) == _declared()


def test_host_side_checks(libsats):
    from paper_2607_08991_gb300 import sats
    L = sats.lib()
    assert L.sats_version() >> 16 == 1
    assert sats.status_string(sats.ESHAPE) == "unsupported shape"
    assert L.sats_workspace_bytes(12, 10, 1) == 0          # H not a multiple of 8
    assert L.sats_workspace_bytes(8, 0, 1) == 0            # N < 1
    assert L.sats_workspace_bytes(16384, 10, 1) == 0       # H too large
    ws = L.sats_workspace_bytes(4096, 14336, 1)
    assert 14336 <= ws <= 14336 + 20480                   # a flag word per 8 neurons + control block, LoRA sums
    assert L.sats_workspace_bytes(4096, 14336, 64) >= ws
    # batches beyond one fused pass run on the tensor cores and need their bf16 staging
    assert L.sats_uses_tensor_cores(4096, 1) == 0 and L.sats_uses_tensor_cores(4096, 2) == 0
    assert L.sats_uses_tensor_cores(4096, 3) == 1 and L.sats_uses_tensor_cores(8192, 2) == 1
    assert L.sats_uses_tensor_cores(512, 2048) == 1
    assert L.sats_workspace_bytes(4096, 14336, 3) >= ws + 3 * (4 * 4096 + 5 * 14336)
    out = ctypes.c_void_p()
    # argument errors come back before any CUDA call
    assert L.sats_layer_create(None, None, None, 64, 64, None, ctypes.byref(out)) == sats.EINVAL
    assert L.sats_layer_create(1, 1, 1, 60, 64, None, ctypes.byref(out)) == sats.ESHAPE
    assert L.sats_layer_create(1, 1, 1, 64, 0, None, None) == sats.EINVAL
    assert L.sats_sparse_mlp(None, None, 1, 0.5, None, None, None, None, 0, None) == sats.EINVAL
    assert L.sats_route(None, 4, None, 10, None, None, None, None) == sats.EINVAL
    assert L.sats_mlp_stack(None, None, None, 1, 1e-5, None, None, 0, None, 1, None, None, 0, None) == sats.EINVAL
    t = ctypes.c_float(-1.0)
    assert L.sats_percentile_threshold(None, 0, 0.5, ctypes.byref(t), None, 0, None) == sats.OK and t.value == 0.0
    assert L.sats_percentile_threshold(None, 10, 0.0, ctypes.byref(t), None, 0, None) == sats.OK and t.value == 0.0
    assert L.sats_percentile_threshold(None, 10, 1.5, ctypes.byref(t), None, 0, None) == sats.OK
    assert t.value == float("inf")


def test_every_entry_rejects_missing_arguments_before_any_cuda_call(libsats):
    """Null pointers and impossible sizes come back as SATS_EINVAL from the host
    checks, with no CUDA call made (this host has no GPU)."""
    from paper_2607_08991_gb300 import sats
    L = sats.lib()
    E = sats.EINVAL
    out = ctypes.c_void_p()
    f, d = ctypes.c_float(), ctypes.c_double()
    assert L.sats_sparse_mlp_f32(None, None, 1, 0.5, None, None, None, None, 0, None) == E
    assert L.sats_sparse_mlp_fixed_scratch(None, None, 1, 0.5, None, None, None, None, None) == E
    assert L.sats_sparse_mlp_union(None, None, 4, 0.5, None, None, None, None, 0, None) == E
    assert L.sats_sparse_mlp_union_f32(None, None, 4, 0.5, None, None, None, None, 0, None) == E
    assert L.sats_lora_create(None, None, None, None, None, None, None, 16, 1.0, None, ctypes.byref(out)) == E
    assert L.sats_sparse_mlp_lora(None, None, None, 1, 0.5, None, None, None, None, 0, None) == E
    assert L.sats_dense_mlp(None, None, 1, None, None, 0, None) == E
    assert L.sats_gate_act(None, None, 1, None, None, 0, None) == E
    assert L.sats_rmsnorm(None, 1, 64, None, 1e-5, None, None) == E
    assert L.sats_layer_err(None, None, 1, None, 1, 1e-6, None, None, None, 0, None) == E
    assert L.sats_token_scores(None, None, None, 10, 100, None, None, 0, None) == E
    assert L.sats_route_calibrate(None, 100, None, 10, 0.5, ctypes.byref(f), ctypes.byref(d), None, None, 0,
                                  None) == E
    assert L.sats_selftest_wait_timeout(None, 0, None) == E
    assert L.sats_selftest_wait_timeout(1, 16, None) == E        # smaller than the control block
    assert L.sats_get_error(None, 0, None) == E
    assert L.sats_get_status_word(None, None) == E
    # the calibration workspaces are host-computed sizes
    assert L.sats_select_workspace_bytes() > 0
    assert L.sats_layer_err_workspace_bytes(4096, 14336, 64, 20) > 0
    assert L.sats_route_calib_workspace_bytes(151936) >= 151936
    assert L.sats_sats_workspace_bytes(4096, 14336, 32, 64, 20, 8) >= L.sats_layer_err_workspace_bytes(4096, 14336,
                                                                                                         64, 20)
