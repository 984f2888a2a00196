"""Python binding of libsats.so (include/sats.h): argument marshalling only.

Every function here forwards to the C ABI of the same name (without the
``sats_`` prefix).  Tensors are torch tensors on the current CUDA device; torch
provides device memory and streams, the library's kernels do every step of the
computation.  There is no fallback: if libsats.so is missing or fails to load,
every call raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libsats.so")

OK, EINVAL, ESHAPE, ECUDA, EDEVICE, ETIMEOUT, ENOSPACE = range(7)

_lib = None


class SatsError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        msg = "%s: %s (status %d)" % (where, status_string(status), status)
        if status == ECUDA:
            msg += ": " + lib().sats_last_cuda_error().decode()
        super().__init__(msg)


def lib() -> ctypes.CDLL:
    """Loads libsats.so (built by paper_2607_08991_gb300.build); raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libsats.so is not built (run __graft_entry__.build()); "
                               "this library has no CPU fallback")
        L = ctypes.CDLL(LIB_PATH)
        P, I, F, D, Z, I64 = (ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_double,
                              ctypes.c_size_t, ctypes.c_int64)
        sig = {
            "sats_version": (I, []),
            "sats_status_string": (ctypes.c_char_p, [I]),
            "sats_layer_create": (I, [P, P, P, I, I, P, ctypes.POINTER(P)]),
            "sats_layer_destroy": (I, [P]),
            "sats_layer_shape": (I, [P, ctypes.POINTER(I), ctypes.POINTER(I)]),
            "sats_workspace_bytes": (Z, [I, I, I]),
            "sats_workspace_init": (I, [P, Z, P]),
            "sats_sparse_mlp": (I, [P, P, I, F, P, P, P, P, Z, P]),
            "sats_sparse_mlp_f32": (I, [P, P, I, F, P, P, P, P, Z, P]),
            "sats_sparse_mlp_fixed_scratch": (I, [P, P, I, F, P, P, P, P, P]),
            "sats_sparse_mlp_union": (I, [P, P, I, F, P, P, P, P, Z, P]),
            "sats_sparse_mlp_union_f32": (I, [P, P, I, F, P, P, P, P, Z, P]),
            "sats_lora_create": (I, [P, P, P, P, P, P, P, I, F, P, ctypes.POINTER(P)]),
            "sats_lora_destroy": (I, [P]),
            "sats_sparse_mlp_lora": (I, [P, P, P, I, F, P, P, P, P, Z, P]),
            "sats_sparse_mlp_lora_f32": (I, [P, P, P, I, F, P, P, P, P, Z, P]),
            "sats_uses_tensor_cores": (I, [I, I]),
            "sats_last_cuda_error": (ctypes.c_char_p, []),
            "sats_dense_mlp": (I, [P, P, I, P, P, Z, P]),
            "sats_route": (I, [P, I, P, I, P, P, P, P]),
            "sats_mlp_stack": (I, [P, P, P, I, F, P, P, I, P, I, P, P, Z, P]),
            "sats_gate_act": (I, [P, P, I, P, P, Z, P]),
            "sats_select_workspace_bytes": (Z, []),
            "sats_percentile_threshold": (I, [P, I64, D, ctypes.POINTER(F), P, Z, P]),
            "sats_rmsnorm": (I, [P, I, I, P, F, P, P]),
            "sats_gate_act_f32": (I, [P, P, I, P, P]),
            "sats_layer_err_workspace_bytes": (Z, [I, I, I, I]),
            "sats_layer_err": (I, [P, P, I, P, I, F, P, P, P, Z, P]),
            "sats_sats_select": (I, [P, P, P, I, I, D, I, D, D, P, P, P]),
            "sats_sats_workspace_bytes": (Z, [I, I, I, I, I, I]),
            "sats_sats_calibrate": (I, [P, P, I, F, P, I, D, I, I, I, F, P, P, P, P, P, P, P, Z, P]),
            "sats_route_calib_workspace_bytes": (Z, [I]),
            "sats_token_scores": (I, [P, P, P, I64, I, P, P, Z, P]),
            "sats_route_calibrate": (I, [P, I, P, I64, D, ctypes.POINTER(F), ctypes.POINTER(D), P, P, Z, P]),
            "sats_get_error": (I, [P, Z, P]),
            "sats_get_status_word": (I, [P, P]),
            "sats_selftest_wait_timeout": (I, [P, Z, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def exported_symbols() -> Sequence[str]:
    """Every C entry point this binding forwards to."""
    return ("sats_version", "sats_status_string", "sats_layer_create", "sats_layer_destroy", "sats_layer_shape",
            "sats_workspace_bytes", "sats_workspace_init", "sats_sparse_mlp", "sats_sparse_mlp_f32",
            "sats_sparse_mlp_fixed_scratch", "sats_sparse_mlp_union", "sats_sparse_mlp_union_f32",
            "sats_lora_create", "sats_lora_destroy", "sats_sparse_mlp_lora", "sats_sparse_mlp_lora_f32",
            "sats_uses_tensor_cores", "sats_last_cuda_error", "sats_dense_mlp", "sats_route", "sats_mlp_stack",
            "sats_gate_act",
            "sats_select_workspace_bytes", "sats_percentile_threshold", "sats_rmsnorm", "sats_gate_act_f32",
            "sats_layer_err_workspace_bytes", "sats_layer_err", "sats_sats_select", "sats_sats_workspace_bytes",
            "sats_sats_calibrate", "sats_route_calib_workspace_bytes", "sats_token_scores", "sats_route_calibrate",
            "sats_get_error", "sats_get_status_word", "sats_selftest_wait_timeout")


def status_string(s: int) -> str:
    return lib().sats_status_string(int(s)).decode()


def _check(s: int, where: str):
    if s != OK:
        raise SatsError(s, where)


def _stream(stream: Optional[torch.cuda.Stream]):
    st = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(st.cuda_stream)


def _ptr(t: Optional[torch.Tensor], name: str, elem: Optional[int] = None):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if elem is not None and t.element_size() != elem:
        raise ValueError("%s must have %d-byte elements" % (name, elem))
    return ctypes.c_void_p(t.data_ptr())


class Layer:
    """Handle of one repacked MLP block (sats_layer_create / sats_layer_destroy)."""

    def __init__(self, W_gate: torch.Tensor, W_up: torch.Tensor, W_down: torch.Tensor,
                 stream: Optional[torch.cuda.Stream] = None):
        H, N = W_gate.shape
        if tuple(W_up.shape) != (H, N) or tuple(W_down.shape) != (N, H):
            raise ValueError("expected W_gate, W_up [H][N] and W_down [N][H]")
        h = ctypes.c_void_p()
        _check(lib().sats_layer_create(_ptr(W_gate, "W_gate", 2), _ptr(W_up, "W_up", 2), _ptr(W_down, "W_down", 2),
                                       H, N, _stream(stream), ctypes.byref(h)), "sats_layer_create")
        self.handle = h
        self.H, self.N = H, N

    def close(self):
        if self.handle is not None and self.handle.value:
            _check(lib().sats_layer_destroy(self.handle), "sats_layer_destroy")
        self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def workspace_bytes(H: int, N: int, B: int) -> int:
    return int(lib().sats_workspace_bytes(H, N, B))


class Workspace:
    """A zero-initialised device workspace (torch memory) for calls up to batch B."""

    def __init__(self, H: int, N: int, B: int, device=None, stream: Optional[torch.cuda.Stream] = None):
        n = workspace_bytes(H, N, B)
        if n == 0:
            raise ValueError("unsupported shape for a workspace: H=%d N=%d B=%d" % (H, N, B))
        self.buf = torch.empty(n, dtype=torch.uint8, device=device or "cuda")
        self.nbytes = n
        _check(lib().sats_workspace_init(_ptr(self.buf, "ws"), n, _stream(stream)), "sats_workspace_init")

    @property
    def ptr(self):
        return ctypes.c_void_p(self.buf.data_ptr())


def sparse_mlp(layer: Layer, x: torch.Tensor, t_l: float, y: torch.Tensor, ws: Workspace,
               active_idx: Optional[torch.Tensor] = None, active_cnt: Optional[torch.Tensor] = None,
               stream: Optional[torch.cuda.Stream] = None):
    B = x.shape[0]
    _check(lib().sats_sparse_mlp(layer.handle, _ptr(x, "x", 2), B, float(t_l), _ptr(y, "y", 4),
                                 _ptr(active_idx, "active_idx", 4), _ptr(active_cnt, "active_cnt", 4),
                                 ws.ptr, ws.nbytes, _stream(stream)), "sats_sparse_mlp")


def sparse_mlp_f32(layer: Layer, x: torch.Tensor, t_l: float, y: torch.Tensor, ws: Workspace,
                   active_idx: Optional[torch.Tensor] = None, active_cnt: Optional[torch.Tensor] = None,
                   stream: Optional[torch.cuda.Stream] = None):
    B = x.shape[0]
    _check(lib().sats_sparse_mlp_f32(layer.handle, _ptr(x, "x", 4), B, float(t_l), _ptr(y, "y", 4),
                                     _ptr(active_idx, "active_idx", 4), _ptr(active_cnt, "active_cnt", 4),
                                     ws.ptr, ws.nbytes, _stream(stream)), "sats_sparse_mlp_f32")


class Lora:
    """A LoRA adapter of one block (sats_lora_create): A_gate, A_up [H][r], B_gate, B_up [r][N],
    A_down [N][r], B_down [r][H] as int16 device tensors of bf16 bit patterns."""

    def __init__(self, layer: Layer, A_gate, B_gate, A_up, B_up, A_down, B_down, scale: float = 1.0,
                 stream: Optional[torch.cuda.Stream] = None):
        r = A_gate.shape[1]
        self.r = r
        out = ctypes.c_void_p()
        _check(lib().sats_lora_create(layer.handle, _ptr(A_gate, "A_gate", 2), _ptr(B_gate, "B_gate", 2),
                                      _ptr(A_up, "A_up", 2), _ptr(B_up, "B_up", 2), _ptr(A_down, "A_down", 2),
                                      _ptr(B_down, "B_down", 2), int(r), float(scale), _stream(stream),
                                      ctypes.byref(out)), "sats_lora_create")
        self.handle = out.value

    def close(self):
        if self.handle:
            _check(lib().sats_lora_destroy(self.handle), "sats_lora_destroy")
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def sparse_mlp_lora(layer: Layer, lora: Lora, x: torch.Tensor, t_l: float, y: torch.Tensor, ws: Workspace,
                    active_idx: Optional[torch.Tensor] = None, active_cnt: Optional[torch.Tensor] = None,
                    stream: Optional[torch.cuda.Stream] = None):
    """sats_sparse_mlp on the adapted weights W + scale A B (x bf16 or fp32)."""
    B = x.shape[0]
    if x.dtype == torch.float32:
        _check(lib().sats_sparse_mlp_lora_f32(layer.handle, lora.handle, _ptr(x, "x", 4), B, float(t_l),
                                              _ptr(y, "y", 4), _ptr(active_idx, "active_idx", 4),
                                              _ptr(active_cnt, "active_cnt", 4), ws.ptr, ws.nbytes,
                                              _stream(stream)), "sats_sparse_mlp_lora_f32")
    else:
        _check(lib().sats_sparse_mlp_lora(layer.handle, lora.handle, _ptr(x, "x", 2), B, float(t_l),
                                          _ptr(y, "y", 4), _ptr(active_idx, "active_idx", 4),
                                          _ptr(active_cnt, "active_cnt", 4), ws.ptr, ws.nbytes, _stream(stream)),
               "sats_sparse_mlp_lora")


def sparse_mlp_union(layer: Layer, x: torch.Tensor, t_l: float, y: torch.Tensor, ws: Workspace,
                     active_idx: Optional[torch.Tensor] = None, active_cnt: Optional[torch.Tensor] = None,
                     stream: Optional[torch.cuda.Stream] = None):
    """sats_sparse_mlp over the union of the batch's kept neurons (x bf16 or fp32; 3 <= B <= 8)."""
    B = x.shape[0]
    if x.dtype == torch.float32:
        _check(lib().sats_sparse_mlp_union_f32(layer.handle, _ptr(x, "x", 4), B, float(t_l), _ptr(y, "y", 4),
                                               _ptr(active_idx, "active_idx", 4), _ptr(active_cnt, "active_cnt", 4),
                                               ws.ptr, ws.nbytes, _stream(stream)), "sats_sparse_mlp_union_f32")
    else:
        _check(lib().sats_sparse_mlp_union(layer.handle, _ptr(x, "x", 2), B, float(t_l), _ptr(y, "y", 4),
                                           _ptr(active_idx, "active_idx", 4), _ptr(active_cnt, "active_cnt", 4),
                                           ws.ptr, ws.nbytes, _stream(stream)), "sats_sparse_mlp_union")


def sparse_mlp_fixed_scratch(layer: Layer, x: torch.Tensor, t_l: float, y: torch.Tensor,
                             active_idx: Optional[torch.Tensor] = None, active_cnt: Optional[torch.Tensor] = None,
                             dev_status: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
    """sats_sparse_mlp without a workspace (the library's fixed 256 KiB device scratch); dev_status, a
    device int32 [1], receives the call's device status word (read it with get_status_word)."""
    B = x.shape[0]
    _check(lib().sats_sparse_mlp_fixed_scratch(layer.handle, _ptr(x, "x", 2), B, float(t_l), _ptr(y, "y", 4),
                                               _ptr(active_idx, "active_idx", 4), _ptr(active_cnt, "active_cnt", 4),
                                               _ptr(dev_status, "dev_status", 4), _stream(stream)),
           "sats_sparse_mlp_fixed_scratch")


def uses_tensor_cores(H: int, B: int) -> bool:
    """True if a batch of B tokens on hidden size H runs on the tensor-core path."""
    return bool(lib().sats_uses_tensor_cores(int(H), int(B)))


def dense_mlp(layer: Layer, x: torch.Tensor, y: torch.Tensor, ws: Workspace,
              stream: Optional[torch.cuda.Stream] = None):
    _check(lib().sats_dense_mlp(layer.handle, _ptr(x, "x", 2), x.shape[0], _ptr(y, "y", 4), ws.ptr, ws.nbytes,
                                _stream(stream)), "sats_dense_mlp")


def route(token_ids: torch.Tensor, lut: torch.Tensor, perm: torch.Tensor, n_dense: torch.Tensor,
          dev_status: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
    _check(lib().sats_route(_ptr(token_ids, "token_ids", 4), token_ids.numel(), _ptr(lut, "lut", 1), lut.numel(),
                            _ptr(perm, "perm", 4), _ptr(n_dense, "n_dense", 4), _ptr(dev_status, "dev_status", 4),
                            _stream(stream)), "sats_route")


def mlp_stack(layers: Sequence[Layer], norm_w: Sequence[torch.Tensor], t: Sequence[float], eps: float,
              x: torch.Tensor, ws: Workspace, token_ids: Optional[torch.Tensor] = None,
              lut: Optional[torch.Tensor] = None, keep_trace: Optional[torch.Tensor] = None,
              stream: Optional[torch.cuda.Stream] = None):
    L = len(layers)
    hs = (ctypes.c_void_p * L)(*[l.handle.value for l in layers])
    nws = (ctypes.c_void_p * L)(*[w.data_ptr() for w in norm_w])
    for w in norm_w:
        _ptr(w, "norm_w", 4)
    ts = (ctypes.c_float * L)(*[float(v) for v in t])
    _check(lib().sats_mlp_stack(hs, nws, ts, L, float(eps), _ptr(token_ids, "token_ids", 4), _ptr(lut, "lut", 1),
                                0 if lut is None else lut.numel(), _ptr(x, "x", 4), x.shape[0],
                                _ptr(keep_trace, "keep_trace", 1), ws.ptr, ws.nbytes, _stream(stream)),
           "sats_mlp_stack")


def gate_act(layer: Layer, x: torch.Tensor, a: torch.Tensor, ws: Optional[Workspace] = None,
             stream: Optional[torch.cuda.Stream] = None):
    _check(lib().sats_gate_act(layer.handle, _ptr(x, "x", 2), x.shape[0], _ptr(a, "a", 4),
                               None if ws is None else ws.ptr, 0 if ws is None else ws.nbytes, _stream(stream)),
           "sats_gate_act")


def select_workspace_bytes() -> int:
    return int(lib().sats_select_workspace_bytes())


def percentile_threshold(a: torch.Tensor, k: float, sel_ws: torch.Tensor,
                         stream: Optional[torch.cuda.Stream] = None) -> float:
    out = ctypes.c_float()
    _check(lib().sats_percentile_threshold(_ptr(a, "a", 4), a.numel(), float(k), ctypes.byref(out),
                                           _ptr(sel_ws, "sel_ws"), sel_ws.numel() * sel_ws.element_size(),
                                           _stream(stream)), "sats_percentile_threshold")
    return float(out.value)


def rmsnorm(x: torch.Tensor, w: torch.Tensor, eps: float, out: torch.Tensor,
            stream: Optional[torch.cuda.Stream] = None):
    B, H = x.shape
    _check(lib().sats_rmsnorm(_ptr(x, "x", 4), B, H, _ptr(w, "w", 4), float(eps), _ptr(out, "out", 4),
                              _stream(stream)), "sats_rmsnorm")


def gate_act_f32(layer: Layer, x: torch.Tensor, a: torch.Tensor, stream: Optional[torch.cuda.Stream] = None):
    _check(lib().sats_gate_act_f32(layer.handle, _ptr(x, "x", 4), x.shape[0], _ptr(a, "a", 4), _stream(stream)),
           "sats_gate_act_f32")


def layer_err(layer: Layer, x: torch.Tensor, t: Sequence[float], eps: float = 1e-6,
              stream: Optional[torch.cuda.Stream] = None):
    """Eq. 6 at each candidate threshold on the calibration inputs x (fp32 [C][H]):
    returns (err, sp) as lists of floats."""
    C = x.shape[0]
    K = len(t)
    n = int(lib().sats_layer_err_workspace_bytes(layer.H, layer.N, C, K))
    ws = torch.empty(n + 256, dtype=torch.uint8, device=x.device)
    off = (-ws.data_ptr()) % 256
    tt = (ctypes.c_float * max(K, 1))(*[float(v) for v in t])
    err = (ctypes.c_double * max(K, 1))()
    sp = (ctypes.c_double * max(K, 1))()
    _check(lib().sats_layer_err(layer.handle, _ptr(x, "x", 4), C, tt, K, float(eps), err, sp,
                                ctypes.c_void_p(ws.data_ptr() + off), n, _stream(stream)), "sats_layer_err")
    return list(err)[:K], list(sp)[:K]


def sats_select(t, err, sp, s_tar: float, guard: int = -1, guard_t: float = 0.0, guard_sp: float = 0.0):
    """Eqs. 7-10 over a [L][K] candidate table (host function): returns (b*, T*(b*), S(b*))."""
    L, K = len(t), len(t[0]) if len(t) else 0
    flat = lambda m: (ctypes.c_double * max(L * K, 1))(*[float(v) for row in m for v in row])
    b = ctypes.c_double()
    S = ctypes.c_double()
    tout = (ctypes.c_double * L)()
    _check(lib().sats_sats_select(flat(t), flat(err), flat(sp), L, K, float(s_tar), int(guard), float(guard_t),
                                  float(guard_sp), ctypes.byref(b), tout, ctypes.byref(S)), "sats_sats_select")
    return b.value, list(tout), S.value


def sats_calibrate(layers: Sequence[Layer], norm_w: Sequence[torch.Tensor], eps: float, x_cal: torch.Tensor,
                   s_tar: float, K0: int = 20, K1: int = 8, guardrail: bool = True, err_eps: float = 1e-6,
                   stream: Optional[torch.cuda.Stream] = None):
    """SATS calibration of a stack (sats_sats_calibrate): returns dict(t, b, S, table=(t, err, sp))."""
    L = len(layers)
    C, H = x_cal.shape
    N = layers[0].N
    n = int(lib().sats_sats_workspace_bytes(H, N, C, L, K0, K1))
    if n == 0:
        raise ValueError("unsupported calibration shape")
    ws = torch.empty(n + 256, dtype=torch.uint8, device=x_cal.device)
    off = (-ws.data_ptr()) % 256
    hs = (ctypes.c_void_p * L)(*[l.handle.value for l in layers])
    nws = (ctypes.c_void_p * L)(*[_ptr(w, "norm_w", 4).value for w in norm_w])
    tout = (ctypes.c_float * L)()
    b = ctypes.c_double()
    S = ctypes.c_double()
    Kt = K0 - 1 + K1
    tt = (ctypes.c_double * (L * Kt))()
    te = (ctypes.c_double * (L * Kt))()
    ts = (ctypes.c_double * (L * Kt))()
    _check(lib().sats_sats_calibrate(hs, nws, L, float(eps), _ptr(x_cal, "x_cal", 4), C, float(s_tar), K0, K1,
                                     1 if guardrail else 0, float(err_eps), tout, ctypes.byref(b), ctypes.byref(S),
                                     tt, te, ts, ctypes.c_void_p(ws.data_ptr() + off), n, _stream(stream)),
           "sats_sats_calibrate")
    rows = lambda arr: [list(arr[l * Kt:(l + 1) * Kt]) for l in range(L)]
    return dict(t=list(tout), b=b.value, S=S.value, table=(rows(tt), rows(te), rows(ts)))


def _calib_ws(V: int, device):
    n = int(lib().sats_route_calib_workspace_bytes(V))
    ws = torch.empty(n + 256, dtype=torch.uint8, device=device)
    return ws, ctypes.c_void_p(ws.data_ptr() + (-ws.data_ptr()) % 256), n


def token_scores(ids: torch.Tensor, l_base: torch.Tensor, l_sparse: torch.Tensor, V: int,
                 stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Eqs. 11-12: per-token mean excess damage (device fp32 [V]; +inf for unseen tokens)."""
    score = torch.empty(V, dtype=torch.float32, device=ids.device)
    keep, ws, n = _calib_ws(V, ids.device)
    _check(lib().sats_token_scores(_ptr(ids, "ids", 4), _ptr(l_base, "l_base", 4), _ptr(l_sparse, "l_sparse", 4),
                                   ids.numel(), V, _ptr(score, "score", 4), ws, n, _stream(stream)),
           "sats_token_scores")
    return score


def route_calibrate(score: torch.Tensor, heldout_ids: torch.Tensor, r_tar: float,
                    stream: Optional[torch.cuda.Stream] = None):
    """Eq. 14: returns (tau*, R(tau*), lut) with lut the device uint8 routing table (1 = base path)."""
    V = score.numel()
    lut = torch.empty(V, dtype=torch.uint8, device=score.device)
    keep, ws, n = _calib_ws(V, score.device)
    tau = ctypes.c_float()
    R = ctypes.c_double()
    _check(lib().sats_route_calibrate(_ptr(score, "score", 4), V, _ptr(heldout_ids, "heldout_ids", 4),
                                      heldout_ids.numel(), float(r_tar), ctypes.byref(tau), ctypes.byref(R),
                                      _ptr(lut, "lut", 1), ws, n, _stream(stream)), "sats_route_calibrate")
    return tau.value, R.value, lut


def selftest_wait_timeout(ws: Workspace, stream: Optional[torch.cuda.Stream] = None):
    """Runs the library's bounded device waits against conditions nothing satisfies; the
    next get_error(ws) reads ETIMEOUT (takes about 4 s)."""
    _check(lib().sats_selftest_wait_timeout(ws.ptr, ws.nbytes, _stream(stream)), "sats_selftest_wait_timeout")


def get_error(ws: Workspace, stream: Optional[torch.cuda.Stream] = None) -> int:
    """Returns the device status of the workspace (OK, EDEVICE or ETIMEOUT) and clears it."""
    return int(lib().sats_get_error(ws.ptr, ws.nbytes, _stream(stream)))


def get_status_word(dev_status: torch.Tensor, stream: Optional[torch.cuda.Stream] = None) -> int:
    return int(lib().sats_get_status_word(_ptr(dev_status, "dev_status", 4), _stream(stream)))
