"""Helpers of the GPU parity tests: device transfer and the comparison rules.

Comparison rules (the tolerance the thresholded path is held to):
  * kept-neuron sets are bit-exact, except neurons whose oracle |a| lies within
    a relative 1e-3 of the threshold (BAND_REL): there either decision is a
    correct result of Eq. 5, and the oracle takes the kernel's decision for
    those neurons only (keep_hint) before computing the expected output;
  * outputs (bf16 weights, fp32 accumulation) against the fp64 oracle on the
    same bf16 values: relative L2 error <= 1e-2 and max-abs error <= 2e-2;
    fp32 arithmetic is held to a tighter relative L2 of 1e-4 as well.
"""
import numpy as np
import torch

BAND_REL = 1e-3
REL_L2 = 1e-2
MAX_ABS = 2e-2
REL_L2_FP32 = 1e-4


def dev_u16(a: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(device)


def dev(a: np.ndarray, device="cuda") -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(a)).to(device)


def keep_from_lists(idx: torch.Tensor, cnt: torch.Tensor, N: int) -> np.ndarray:
    idx = idx.cpu().numpy()
    cnt = cnt.cpu().numpy()
    keep = np.zeros((idx.shape[0], N), np.uint8)
    for b in range(idx.shape[0]):
        lst = idx[b, : cnt[b]]
        assert np.all(np.diff(lst) > 0), "active list not strictly increasing"
        assert lst.size == 0 or (lst[0] >= 0 and lst[-1] < N)
        keep[b, lst] = 1
    return keep


def band_mask(a_ref: np.ndarray, t) -> np.ndarray:
    t = np.broadcast_to(np.asarray(t, np.float64), (a_ref.shape[0],))[:, None]
    return np.isfinite(t) & (np.abs(np.abs(a_ref) - t) <= BAND_REL * t)


def assert_keep_match(keep_gpu: np.ndarray, keep_ref: np.ndarray, a_ref: np.ndarray, t):
    band = band_mask(a_ref, t)
    diff = (keep_gpu != keep_ref) & ~band
    assert not diff.any(), "kept sets differ outside the threshold band at %s" % (np.argwhere(diff)[:5].tolist(),)


def assert_close(y_gpu, y_ref, tight: bool = True):
    y_gpu = np.asarray(y_gpu, np.float64)
    y_ref = np.asarray(y_ref, np.float64)
    assert y_gpu.shape == y_ref.shape
    assert np.all(np.isfinite(y_gpu))
    nref = np.linalg.norm(y_ref)
    err = np.linalg.norm(y_gpu - y_ref)
    rel = err / nref if nref > 0 else err
    mx = np.abs(y_gpu - y_ref).max() if y_ref.size else 0.0
    assert rel <= REL_L2, "relative L2 error %.3e" % rel
    assert mx <= MAX_ABS, "max abs error %.3e" % mx
    if tight:
        assert rel <= REL_L2_FP32, "relative L2 error %.3e above the fp32 bound" % rel
    return rel, mx
