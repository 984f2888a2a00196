"""CPU oracle for the thresholded gated MLP and token routing (test infrastructure).

This package is TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()``
and the ``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import
it.  It shares no code with the CUDA library in ``paper_2607_08991_gb300``:
the MLP arithmetic (Sec. 2, Eqs. 1-5), Eq. 3, routing (Eq. 13), the stack,
Eq. 6 and Eqs. 7-10 live in ``sats_oracle.c`` (plain C, IEEE double),
compiled with gcc into ``liboracle.so`` and called through ctypes; the
routing calibration (Sec. 3.2, Eqs. 11-14) and the order of the SATS
coarse-to-fine steps are written out here in numpy (float64).

Paper: "Sensitivity-Aware Thresholding and Token Routing for Activation
Sparsification in Large Language Models" (arXiv 2607.08991).  Each wrapper
names the section / equation its C routine states.

Parity status: every function here is pinned by ``tests/test_oracle_*.py``
(closed forms, brute force on tiny inputs, library cross-checks and
invariants).  No function is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sats_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile sats_oracle.c into liboracle.so with gcc (portable flags only)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + ".tmp.%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        I = ctypes.c_int
        I64 = ctypes.c_int64
        D = ctypes.c_double
        lib.oracle_bf16_to_f64.argtypes = [I64, P, P]
        lib.oracle_silu.argtypes = [D]
        lib.oracle_silu.restype = D
        lib.oracle_gate_act.argtypes = [I, I, I, P, P, P]
        lib.oracle_up_proj.argtypes = [I, I, I, P, P, P]
        lib.oracle_cats_mask.argtypes = [I, I, P, P, P, D, P]
        lib.oracle_cats_mask.restype = I64
        lib.oracle_masked_mlp.argtypes = [I, I, I, P, P, P, P, P, P]
        lib.oracle_sparse_mlp.argtypes = [I, I, I, P, P, P, P, P, P, D, P, P, P]
        lib.oracle_sparse_mlp.restype = I64
        lib.oracle_sparse_mlp_lora.argtypes = [I, I, I, I, P, P, P, P, P, P, P, P, P, P, D, P, P, D, P, P, P]
        lib.oracle_sparse_mlp_lora.restype = I64
        lib.oracle_dense_mlp.argtypes = [I, I, I, P, P, P, P, P]
        lib.oracle_percentile_threshold.argtypes = [P, I64, D]
        lib.oracle_percentile_threshold.restype = D
        lib.oracle_route.argtypes = [I, P, I, P, P, P]
        lib.oracle_route.restype = I
        lib.oracle_rmsnorm.argtypes = [I, I, P, P, D, P]
        lib.oracle_mlp_stack.argtypes = [I, I, I, I, P, P, P, P, P, D, P, P, I, P, P, D, P]
        lib.oracle_mlp_stack.restype = I64
        lib.oracle_layer_err.argtypes = [I, I, I, P, P, P, P, I, P, D, P, P]
        lib.oracle_sats_select.argtypes = [I, I, P, P, P, D, I, D, D, P, P, P]
        _lib = lib
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _u16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    assert a.dtype == np.uint16, "weights are bf16 bit patterns (uint16)"
    return a


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of each bf16 bit pattern, as float64."""
    bits = _u16(bits)
    out = np.empty(bits.shape, dtype=np.float64)
    _load().oracle_bf16_to_f64(bits.size, _ptr(bits), _ptr(out))
    return out


def silu(z: float) -> float:
    """Sec. 2, Eq. 2."""
    return _load().oracle_silu(float(z))


def gate_act(x: np.ndarray, Wg: np.ndarray) -> np.ndarray:
    """Sec. 2, Eqs. 1-2: SiLU(x W_gate); x [B][H] float64, Wg [H][N] bf16 bits."""
    x = _f64(x)
    Wg = _u16(Wg)
    B, H = x.shape
    N = Wg.shape[1]
    a = np.empty((B, N), dtype=np.float64)
    _load().oracle_gate_act(B, H, N, _ptr(x), _ptr(Wg), _ptr(a))
    return a


def up_proj(x: np.ndarray, Wu: np.ndarray) -> np.ndarray:
    """Sec. 2, Eq. 1: x W_up."""
    x = _f64(x)
    Wu = _u16(Wu)
    B, H = x.shape
    N = Wu.shape[1]
    u = np.empty((B, N), dtype=np.float64)
    _load().oracle_up_proj(B, H, N, _ptr(x), _ptr(Wu), _ptr(u))
    return u


def cats_mask(a: np.ndarray, t, keep_hint: Optional[np.ndarray] = None, band_rel: float = 0.0):
    """Sec. 2, Eqs. 4-5: keep iff |a| >= t.  Returns (keep uint8 [B][N], in_band)."""
    a = _f64(a)
    B, N = a.shape
    tt = _f64(np.broadcast_to(np.asarray(t, dtype=np.float64), (B,)))
    keep = np.empty((B, N), dtype=np.uint8)
    hint = None if keep_hint is None else np.ascontiguousarray(keep_hint, dtype=np.uint8)
    nb = _load().oracle_cats_mask(B, N, _ptr(a), _ptr(tt), _ptr(hint), float(band_rel), _ptr(keep))
    return keep, int(nb)


def masked_mlp(x, Wg, Wu, Wd, keep) -> np.ndarray:
    """Sec. 2, Eqs. 1 and 5 with a given mask."""
    x = _f64(x)
    Wg, Wu, Wd = _u16(Wg), _u16(Wu), _u16(Wd)
    B, H = x.shape
    N = Wg.shape[1]
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    y = np.empty((B, H), dtype=np.float64)
    _load().oracle_masked_mlp(B, H, N, _ptr(x), _ptr(Wg), _ptr(Wu), _ptr(Wd), _ptr(keep), _ptr(y))
    return y


def sparse_mlp(x, Wg, Wu, Wd, t, keep_hint=None, band_rel: float = 0.0):
    """Sec. 2, Eqs. 1-5: the CATS-thresholded gated MLP with per-token threshold t.

    Returns (y [B][H] float64, a [B][N] float64, keep [B][N] uint8, in_band).
    """
    x = _f64(x)
    Wg, Wu, Wd = _u16(Wg), _u16(Wu), _u16(Wd)
    B, H = x.shape
    N = Wg.shape[1]
    assert Wg.shape == (H, N) and Wu.shape == (H, N) and Wd.shape == (N, H)
    tt = _f64(np.broadcast_to(np.asarray(t, dtype=np.float64), (B,)))
    hint = None if keep_hint is None else np.ascontiguousarray(keep_hint, dtype=np.uint8)
    y = np.empty((B, H), dtype=np.float64)
    a = np.empty((B, N), dtype=np.float64)
    keep = np.empty((B, N), dtype=np.uint8)
    nb = _load().oracle_sparse_mlp(B, H, N, _ptr(x), _ptr(Wg), _ptr(Wu), _ptr(Wd), _ptr(tt),
                                   _ptr(hint), float(band_rel), _ptr(y), _ptr(a), _ptr(keep))
    return y, a, keep, int(nb)


def sparse_mlp_lora(x, Wg, Wu, Wd, lora, scale: float, t, keep_hint=None, band_rel: float = 0.0):
    """Sec. 4 (fine-tuned routing): the sparse path on LoRA-adapted projections
    W + scale A B, the low-rank terms applied factor by factor (Sec. 2, Eqs. 1-5
    otherwise).  lora = (Ag [H][r], Bg [r][N], Au [H][r], Bu [r][N], Ad [N][r],
    Bd [r][H]) as bf16 bit patterns.  Returns (y, a, keep, in_band) as sparse_mlp."""
    x = _f64(x)
    Wg, Wu, Wd = _u16(Wg), _u16(Wu), _u16(Wd)
    Ag, Bg, Au, Bu, Ad, Bd = (_u16(m) for m in lora)
    B, H = x.shape
    N = Wg.shape[1]
    r = Ag.shape[1]
    assert Ag.shape == (H, r) and Au.shape == (H, r) and Bg.shape == (r, N) and Bu.shape == (r, N)
    assert Ad.shape == (N, r) and Bd.shape == (r, H)
    tt = _f64(np.broadcast_to(np.asarray(t, dtype=np.float64), (B,)))
    hint = None if keep_hint is None else np.ascontiguousarray(keep_hint, dtype=np.uint8)
    y = np.empty((B, H), dtype=np.float64)
    a = np.empty((B, N), dtype=np.float64)
    keep = np.empty((B, N), dtype=np.uint8)
    nb = _load().oracle_sparse_mlp_lora(B, H, N, r, _ptr(x), _ptr(Wg), _ptr(Wu), _ptr(Wd), _ptr(Ag), _ptr(Bg),
                                        _ptr(Au), _ptr(Bu), _ptr(Ad), _ptr(Bd), float(scale), _ptr(tt),
                                        _ptr(hint), float(band_rel), _ptr(y), _ptr(a), _ptr(keep))
    return y, a, keep, int(nb)


def dense_mlp(x, Wg, Wu, Wd) -> np.ndarray:
    """Sec. 2, Eq. 1: the base gated MLP, no mask."""
    x = _f64(x)
    Wg, Wu, Wd = _u16(Wg), _u16(Wu), _u16(Wd)
    B, H = x.shape
    N = Wg.shape[1]
    y = np.empty((B, H), dtype=np.float64)
    _load().oracle_dense_mlp(B, H, N, _ptr(x), _ptr(Wg), _ptr(Wu), _ptr(Wd), _ptr(y))
    return y


def percentile_threshold(values: np.ndarray, k: float) -> float:
    """Sec. 2, Eq. 3: t = min{t' : F(t') >= k} over the magnitudes of `values`."""
    v = _f64(values).ravel()
    return float(_load().oracle_percentile_threshold(_ptr(v), v.size, float(k)))


def route(ids: np.ndarray, lut: np.ndarray):
    """Sec. 3.2, Eq. 13 as a LUT: returns (perm int32 [B], n_dense) or raises on a bad id."""
    ids = np.ascontiguousarray(ids, dtype=np.int32)
    lut = np.ascontiguousarray(lut, dtype=np.uint8)
    B = ids.size
    perm = np.empty(max(B, 1), dtype=np.int32)
    nd = np.zeros(1, dtype=np.int32)
    rc = _load().oracle_route(B, _ptr(ids), lut.size, _ptr(lut), _ptr(perm), _ptr(nd))
    if rc != 0:
        raise ValueError("token id outside the vocabulary")
    return perm[:B].copy(), int(nd[0])


def rmsnorm(x, w, eps: float) -> np.ndarray:
    x = _f64(x)
    B, H = x.shape
    w = np.ascontiguousarray(w, dtype=np.float32)
    out = np.empty_like(x)
    _load().oracle_rmsnorm(B, H, _ptr(x), _ptr(w), float(eps), _ptr(out))
    return out


def mlp_stack(x, Wg: Sequence, Wu: Sequence, Wd: Sequence, norm_w: Sequence, t, eps: float,
              ids=None, lut=None, keep_hint=None, band_rel: float = 0.0, want_keep: bool = False):
    """Stack of L RMSNorm -> gated MLP -> residual blocks with per-token routing.

    Returns (x_out [B][H] float64, keep [L][B][N] uint8 or None, in_band).
    """
    x = _f64(x).copy()
    B, H = x.shape
    L = len(Wg)
    N = Wg[0].shape[1]
    keep_ref = [_u16(w) for w in Wg], [_u16(w) for w in Wu], [_u16(w) for w in Wd]
    nw = [np.ascontiguousarray(w, dtype=np.float32) for w in norm_w]
    arr = lambda lst: (ctypes.c_void_p * L)(*[a.ctypes.data for a in lst])
    tt = _f64(np.broadcast_to(np.asarray(t, dtype=np.float64), (L,)))
    if ids is not None:
        ids_a = np.ascontiguousarray(ids, dtype=np.int32)
        lut_a = np.ascontiguousarray(lut, dtype=np.uint8)
        V = lut_a.size
    else:
        ids_a = lut_a = None
        V = 0
    hint = None if keep_hint is None else np.ascontiguousarray(keep_hint, dtype=np.uint8)
    keep = np.empty((L, B, N), dtype=np.uint8) if want_keep else None
    nb = _load().oracle_mlp_stack(L, B, H, N, arr(keep_ref[0]), arr(keep_ref[1]), arr(keep_ref[2]),
                                  arr(nw), _ptr(tt), float(eps), _ptr(ids_a), _ptr(lut_a), V,
                                  _ptr(x), _ptr(hint), float(band_rel), _ptr(keep))
    if nb < 0:
        raise ValueError("token id outside the vocabulary")
    return x, keep, int(nb)


def layer_err(x, Wg, Wu, Wd, t, eps: float = 1e-6):
    """Sec. 3.1, Eq. 6 at each candidate threshold t[k] on the calibration inputs x [C][H]
    (the block's MLP inputs).  Returns (err [K], sp [K]): the mean relative L2 distortion
    ||y - y~_t|| / (||y|| + eps) and the mean fraction of neurons with |a| < t."""
    x = _f64(x)
    Wg, Wu, Wd = _u16(Wg), _u16(Wu), _u16(Wd)
    C, H = x.shape
    N = Wg.shape[1]
    t = _f64(np.atleast_1d(t))
    err = np.empty(t.size, dtype=np.float64)
    sp = np.empty(t.size, dtype=np.float64)
    _load().oracle_layer_err(C, H, N, _ptr(x), _ptr(Wg), _ptr(Wu), _ptr(Wd), t.size, _ptr(t), float(eps),
                             _ptr(err), _ptr(sp))
    return err, sp


def sats_select(t, err, sp, s_tar: float, guard: int = -1, guard_t: float = 0.0, guard_sp: float = 0.0):
    """Sec. 3.1, Eqs. 7-10 over a candidate table t, err, sp of shape [L][K].
    Returns (b*, T*(b*) [L], S(b*))."""
    t, err, sp = _f64(t), _f64(err), _f64(sp)
    L, K = t.shape
    assert err.shape == (L, K) and sp.shape == (L, K)
    b = np.zeros(1)
    S = np.zeros(1)
    tout = np.empty(L, dtype=np.float64)
    _load().oracle_sats_select(L, K, _ptr(t), _ptr(err), _ptr(sp), float(s_tar), int(guard), float(guard_t),
                               float(guard_sp), _ptr(b), _ptr(tout), _ptr(S))
    return float(b[0]), tout, float(S[0])


def sats_calibrate(x_cal, Wg: Sequence, Wu: Sequence, Wd: Sequence, norm_w: Sequence, eps: float, s_tar: float,
                   K0: int = 20, K1: int = 8, guardrail: bool = True, err_eps: float = 1e-6):
    """SATS calibration of a stack (Sec. 3.1, Eqs. 3, 6-10, coarse-to-fine; Sec. 4 guardrail),
    in the paper's order:

    1. the dense stack on the calibration inputs gives each block's MLP inputs
       n_l = RMSNorm(x_l) w_l, with x_{l+1} = x_l + MLP_l(n_l);
    2. coarse candidates T_l: Eq. 3 percentiles of |SiLU(n_l W_gate)| at k / K0, k = 1 .. K0-1;
    3. Err_l(t) and sp_l(t) for every candidate (Eq. 6);
    4. b* and T*(b*) (Eqs. 7-10); with the guardrail the last block keeps the CATS
       threshold at s_tar (its Eq. 3 percentile);
    5. fine candidates: K1 thresholds evenly spaced strictly between the coarse candidates
       that neighbour t*_l (0 below the first; the largest |a| above the last);
    6. Eqs. 6-10 again over coarse and fine candidates together.

    Returns dict(t [L], b, S, coarse=(t, err, sp), fine=(t, err, sp) [L][K0-1+K1])."""
    x = _f64(x_cal).copy()
    L = len(Wg)
    inputs_l, amax, guard = [], [], (L - 1 if guardrail else -1)
    cand = np.zeros((L, K0 - 1))
    for l in range(L):
        n = rmsnorm(x, norm_w[l], eps)
        inputs_l.append(n)
        a = gate_act(n, Wg[l])
        amax.append(float(np.abs(a).max()))
        cand[l] = [percentile_threshold(a, k / K0) for k in range(1, K0)]
        x = x + dense_mlp(n, Wg[l], Wu[l], Wd[l])
    err0 = np.zeros_like(cand)
    sp0 = np.zeros_like(cand)
    for l in range(L):
        err0[l], sp0[l] = layer_err(inputs_l[l], Wg[l], Wu[l], Wd[l], cand[l], err_eps)
    g_t = g_sp = 0.0
    if guard >= 0:
        g_t = percentile_threshold(gate_act(inputs_l[guard], Wg[guard]), s_tar)
        g_sp = float(layer_err(inputs_l[guard], Wg[guard], Wu[guard], Wd[guard], [g_t], err_eps)[1][0])
    b0, t0, _ = sats_select(cand, err0, sp0, s_tar, guard, g_t, g_sp)
    fine = np.zeros((L, K1))
    for l in range(L):
        below = cand[l][cand[l] < t0[l]]
        above = cand[l][cand[l] > t0[l]]
        lo = below.max() if below.size else 0.0
        hi = above.min() if above.size else amax[l]
        fine[l] = lo + (hi - lo) * np.arange(1, K1 + 1) / (K1 + 1)
    err1 = np.zeros_like(fine)
    sp1 = np.zeros_like(fine)
    for l in range(L):
        err1[l], sp1[l] = layer_err(inputs_l[l], Wg[l], Wu[l], Wd[l], fine[l], err_eps)
    t_all = np.concatenate([cand, fine], axis=1)
    e_all = np.concatenate([err0, err1], axis=1)
    s_all = np.concatenate([sp0, sp1], axis=1)
    b, t, S = sats_select(t_all, e_all, s_all, s_tar, guard, g_t, g_sp)
    return dict(t=t, b=b, S=S, coarse=(cand, err0, sp0), fine=(t_all, e_all, s_all), guard=(g_t, g_sp))


# ---------------------------------------------------------------- routing calibration (Sec. 3.2)

def token_scores(ids, l_base, l_sparse, V: int) -> np.ndarray:
    """Sec. 3.2, Eqs. 11-12: d_i = max(0, l_sparse_i - l_base_i) for every corpus occurrence i,
    and s(x) = the mean of d_i over I_x = {i : x_i = x}.  A token with no occurrence has no
    estimate; it gets +inf (the base path under Eq. 13 for every tau).  Raises on an id outside [0, V)."""
    ids = np.asarray(ids, dtype=np.int64)
    if ids.size and (ids.min() < 0 or ids.max() >= V):
        raise ValueError("token id outside the vocabulary")
    d = np.maximum(0.0, np.asarray(l_sparse, np.float64) - np.asarray(l_base, np.float64))   # Eq. 11
    total = np.bincount(ids, weights=d, minlength=V)
    count = np.bincount(ids, minlength=V)
    s = np.full(V, np.inf)
    seen = count > 0
    s[seen] = total[seen] / count[seen]                                                      # Eq. 12
    return s


def routed_fraction(score, heldout_ids, tau) -> float:
    """R(tau): the fraction of held-out occurrences routed to the sparse path, score < tau (Eq. 13)."""
    s = np.asarray(score, np.float64)[np.asarray(heldout_ids, np.int64)]
    return float(np.mean(s < tau)) if s.size else 0.0


def route_threshold(score, heldout_ids, r_tar: float):
    """Sec. 3.2, Eq. 14: tau* = argmin_tau |R(tau) - r_tar| over the candidates 0, every score of a
    token occurring in the held-out split, and +inf (R only changes at those values); a tie goes to
    the smaller tau.  Returns (tau*, R(tau*))."""
    s = np.sort(np.asarray(score, np.float64)[np.asarray(heldout_ids, np.int64)])
    cands = np.unique(np.concatenate([[0.0], s[np.isfinite(s)], [np.inf]]))
    R = np.searchsorted(s, cands, side="left") / max(s.size, 1)
    gaps = np.abs(R - r_tar)
    k = int(np.argmin(gaps))          # first minimum: the smallest tau among ties
    return float(cands[k]), float(R[k])


def route_lut(score, tau: float) -> np.ndarray:
    """Eq. 13 as a table: 1 (base path) where score >= tau, 0 (sparse path) where score < tau."""
    return (np.asarray(score, np.float64) >= tau).astype(np.uint8)
