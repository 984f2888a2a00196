"""Seeded synthetic inputs shared by the tests, the bench and the oracle checks.

This module only draws random numbers and packs them into the bit layouts the
two sides take (bf16 bit patterns as uint16, fp32, int32, uint8).  It holds
none of the method's arithmetic: no projection, activation, threshold,
percentile or routing rule.  Thresholds are chosen by the method's own
calibration routine on each side (Eq. 3 of arXiv 2607.08991).

Shapes and distributions follow the workloads the paper runs on
(Llama-3.1-8B: hidden 4096, intermediate 14336, vocab 128256, 32 blocks;
Qwen3-8B: hidden 4096, intermediate 12288, vocab 151936, 36 blocks), with
synthetic weights ~ N(0, 0.02) in bf16 standing in for the trained weights.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List

import numpy as np

LLAMA_H, LLAMA_N, LLAMA_L, LLAMA_V = 4096, 14336, 32, 128256
QWEN_H, QWEN_N, QWEN_L, QWEN_V = 4096, 12288, 36, 151936
SMALL_H, SMALL_N = 512, 1408

# Seed bases: weights of layer l use SEED_WEIGHTS + l (gate / up / down are
# sub-streams 0 / 1 / 2), evaluation activations SEED_X, calibration
# activations SEED_CALIB, routing table SEED_LUT, token ids SEED_IDS,
# RMSNorm weights SEED_NORM + l.
SEED_WEIGHTS = 1000
SEED_X = 2000
SEED_CALIB = 3000
SEED_LUT = 4000
SEED_IDS = 5000
SEED_NORM = 6000
SEED_SHUFFLE = 7000


def _rng(*seed: int) -> np.random.Generator:
    return np.random.default_rng(list(seed))


def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); returns uint16 bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    r = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float32 (exact)."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal_bf16(shape, std: float, *seed: int) -> np.ndarray:
    z = _rng(*seed).standard_normal(size=shape, dtype=np.float32)
    z *= np.float32(std)
    return to_bf16_bits(z)


@dataclasses.dataclass
class MLPWeights:
    """One gated-MLP block in the paper's layout: Wg, Wu [H][N]; Wd [N][H] (bf16 bits)."""
    Wg: np.ndarray
    Wu: np.ndarray
    Wd: np.ndarray

    @property
    def H(self) -> int:
        return self.Wg.shape[0]

    @property
    def N(self) -> int:
        return self.Wg.shape[1]


def mlp_weights(H: int, N: int, layer: int = 0, std: float = 0.02, seed: int = SEED_WEIGHTS) -> MLPWeights:
    return MLPWeights(
        Wg=normal_bf16((H, N), std, seed + layer, 0),
        Wu=normal_bf16((H, N), std, seed + layer, 1),
        Wd=normal_bf16((N, H), std, seed + layer, 2),
    )


def _seed63(*seed: int) -> int:
    return int(np.random.SeedSequence(list(seed)).generate_state(1, np.uint64)[0] & np.uint64((1 << 63) - 1))


def device_normal_bf16(shape, std: float, *seed: int, device="cuda"):
    """N(0, std) rounded to bf16 (nearest even), drawn on a CUDA device by torch's
    seeded Philox generator: a device int16 tensor of bf16 bit patterns.  For
    the model-sized weights of the full-size workloads, which the host would
    take minutes to draw; the oracle gets the same values by copying them to
    the host (`host_bits`)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(_seed63(*seed))
    z = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    z.mul_(std)
    return z.to(torch.bfloat16).view(torch.int16)


def host_bits(t) -> np.ndarray:
    """A device int16 tensor of bf16 bit patterns -> uint16 numpy array on the host."""
    return t.cpu().numpy().view(np.uint16)


def mlp_weights_device(H: int, N: int, layer: int = 0, std: float = 0.02, seed: int = SEED_WEIGHTS,
                       device="cuda"):
    """The weights of layer `layer` drawn on the device: (Wg [H][N], Wu [H][N], Wd [N][H]) int16 tensors."""
    return (device_normal_bf16((H, N), std, seed + layer, 10, device=device),
            device_normal_bf16((H, N), std, seed + layer, 11, device=device),
            device_normal_bf16((N, H), std, seed + layer, 12, device=device))


def lora_adapter(H: int, N: int, r: int, std_a: float = 0.02, std_b: float = 0.02, seed: int = 7000,
                 layer: int = 0):
    """A synthetic LoRA adapter of rank r for one MLP block (the trained adapters are not
    available): (Ag [H][r], Bg [r][N], Au [H][r], Bu [r][N], Ad [N][r], Bd [r][H]), every
    factor N(0, std) rounded to bf16 (bit patterns).  Unlike LoRA's zero-initialised B,
    both factors are non-zero so that every low-rank term is exercised."""
    return (normal_bf16((H, r), std_a, seed + layer, 20), normal_bf16((r, N), std_b, seed + layer, 21),
            normal_bf16((H, r), std_a, seed + layer, 22), normal_bf16((r, N), std_b, seed + layer, 23),
            normal_bf16((N, r), std_a, seed + layer, 24), normal_bf16((r, H), std_b, seed + layer, 25))


def activations_bf16(B: int, H: int, seed: int = SEED_X) -> np.ndarray:
    """x ~ N(0, 1) rounded to bf16: [B][H] uint16 bit patterns."""
    return normal_bf16((B, H), 1.0, seed)


def activations_correlated_bf16(B: int, H: int, rho: float, seed: int = SEED_X) -> np.ndarray:
    """x_m = rho z_0 + sqrt(1 - rho^2) z_m with z ~ N(0, 1) i.i.d. (so every x_m is
    N(0, 1) and any two tokens correlate with coefficient rho^2 elementwise),
    rounded to bf16: [B][H] uint16 bit patterns.  A stand-in for batches whose
    tokens share most of their kept neurons."""
    z = _rng(seed, 2).standard_normal(size=(B + 1, H))
    x = rho * z[0] + np.sqrt(1.0 - rho * rho) * z[1:]
    return to_bf16_bits(x.astype(np.float32))


def activations_f32(B: int, H: int, seed: int = SEED_X) -> np.ndarray:
    return _rng(seed, 1).standard_normal(size=(B, H), dtype=np.float32)


def norm_weight(H: int, layer: int = 0, seed: int = SEED_NORM) -> np.ndarray:
    """RMSNorm gain 1 + N(0, 0.02), float32 [H]."""
    return (1.0 + 0.02 * _rng(seed + layer).standard_normal(size=H)).astype(np.float32)


def routing_lut(V: int, p_dense: float, seed: int = SEED_LUT) -> np.ndarray:
    """Bernoulli(p_dense) table over the vocabulary; 1 = base (dense) path."""
    return (_rng(seed).random(V) < p_dense).astype(np.uint8)


def token_ids_uniform(B: int, V: int, seed: int = SEED_IDS) -> np.ndarray:
    return _rng(seed).integers(0, V, size=B, dtype=np.int64).astype(np.int32)


def token_ids_zipf(B: int, V: int, s: float = 1.1, seed: int = SEED_IDS) -> np.ndarray:
    """Zipf(s) truncated to V ranks via its explicit CDF; rank r -> token id r-1."""
    ranks = np.arange(1, V + 1, dtype=np.float64)
    p = ranks ** (-s)
    cdf = np.cumsum(p)
    cdf /= cdf[-1]
    u = _rng(seed).random(B)
    return np.minimum(np.searchsorted(cdf, u, side="right"), V - 1).astype(np.int32)


def routing_corpus(n: int, V: int, seed: int = SEED_IDS + 100, s: float = 1.1):
    """A synthetic stand-in for the routing calibration corpus of Sec. 3.2: n token
    occurrences with Zipf(s) ids over V, a base-path loss l_base ~ N(3, 1), and a
    sparse-path loss l_sparse = l_base + r(x) + N(0, 0.05), where r(v) ~ Exp(0.1) is a
    per-token risk (so the excess damage depends on the token, as the method assumes).
    Returns (ids int32 [n], l_base fp32 [n], l_sparse fp32 [n])."""
    ids = token_ids_zipf(n, V, s=s, seed=seed)
    g = _rng(seed, 1)
    risk = g.exponential(0.1, size=V).astype(np.float32)
    l_base = (3.0 + g.standard_normal(n)).astype(np.float32)
    l_sparse = (l_base + risk[ids] + 0.05 * g.standard_normal(n)).astype(np.float32)
    return ids, l_base, l_sparse


def stack_sparsity_targets(L: int, lo: float, hi: float, seed: int = SEED_SHUFFLE) -> np.ndarray:
    """L evenly spaced targets in [lo, hi] (mean (lo+hi)/2), assigned to layers by a seeded shuffle."""
    base = lo + (hi - lo) * (np.arange(L) + 0.5) / L
    return base[_rng(seed).permutation(L)]


# The five workloads, by what they are.
WORKLOADS: Dict[str, dict] = {
    "small_layer_512x1408_b1": dict(H=SMALL_H, N=SMALL_N, B=1, calib=64, sparsity=[0.5]),
    "llama_layer_4096x14336_b1": dict(H=LLAMA_H, N=LLAMA_N, B=1, calib=256, sparsity=[0.5, 0.7, 0.9]),
    "llama_stack_32x4096x14336_b1x128": dict(H=LLAMA_H, N=LLAMA_N, L=LLAMA_L, B=1, tokens=128,
                                            sparsity_range=(0.55, 0.85), eps=1e-5),
    "qwen_stack_36x4096x12288_routed": dict(H=QWEN_H, N=QWEN_N, L=QWEN_L, V=QWEN_V, batches=[1, 8, 32, 64],
                                           p_dense=0.3, sparsity=0.5, eps=1e-6),
    "llama_layer_prefill_routed": dict(H=LLAMA_H, N=LLAMA_N, V=LLAMA_V, batches=[256, 2048], zipf_s=1.1,
                                       p_dense=0.2, sparsity=[0.4, 0.6, 0.8, 0.9]),
    # routing calibration (Sec. 3.2) over the Qwen3-8B-shaped vocabulary
    "route_calibration_qwen_v151936": dict(V=QWEN_V, corpus=4_000_000, heldout=1_000_000,
                                           targets=[0.25, 0.5, 0.75]),
    # batched decode on the union of the kept neurons, independent and correlated tokens
    "union_batch_llama_4096x14336": dict(H=LLAMA_H, N=LLAMA_N, batches=[3, 4, 8], sparsity=[0.7, 0.9],
                                         rho=[0.0, 0.9], calib=256),
    # the LoRA-aware sparse path (Sec. 4, fine-tuned routing) on the Llama layer, one decode token
    "lora_llama_layer_4096x14336_b1": dict(H=LLAMA_H, N=LLAMA_N, ranks=[16, 32], sparsity=[0.5, 0.7, 0.9],
                                           calib=256, scale=1.0),
    # SATS calibration (Sec. 3.1) of the 32-block Llama-shaped stack
    "sats_calibration_llama_32x4096x14336": dict(H=LLAMA_H, N=LLAMA_N, L=LLAMA_L, calib=64, K0=20, K1=8,
                                                  target=0.5, eps=1e-5),
}
