"""The seeded input generators (paper_2607_08991_gb300/inputs.py), which both the
oracle's tests and the CUDA path's tests draw from: deterministic per seed, bf16
rounding to nearest even (checked against torch's own conversion), the requested
distributions, and the synthetic workload recipes as stated (the stack's sparsity
targets, Zipf token ids, correlated batches)."""
import math

import numpy as np
import torch

from paper_2607_08991_gb300 import inputs


def test_same_seed_same_values_other_seed_other_values():
    a, b, c = (inputs.mlp_weights(16, 24, seed=s) for s in (5, 5, 6))
    for m in ("Wg", "Wu", "Wd"):
        assert np.array_equal(getattr(a, m), getattr(b, m))
        assert not np.array_equal(getattr(a, m), getattr(c, m))
    assert not np.array_equal(a.Wg, a.Wu)   # the three matrices draw from their own streams
    for f in (lambda s: inputs.activations_bf16(3, 64, seed=s), lambda s: inputs.activations_f32(3, 64, seed=s),
              lambda s: inputs.routing_lut(1000, 0.3, seed=s), lambda s: inputs.token_ids_zipf(100, 1000, seed=s),
              lambda s: inputs.stack_sparsity_targets(32, 0.55, 0.85, seed=s),
              lambda s: np.concatenate([m.ravel() for m in inputs.lora_adapter(16, 24, 4, seed=s)])):
        assert np.array_equal(f(11), f(11))
        assert not np.array_equal(f(11), f(12))


def test_bf16_rounding_is_nearest_even():
    one = np.float32(1.0)
    cases = {
        1.0: 0x3F80,
        1.0 + 2.0 ** -8: 0x3F80,                 # halfway between 0x3F80 and 0x3F81: to the even one
        1.0 + 3 * 2.0 ** -8: 0x3F82,             # halfway between 0x3F81 and 0x3F82: to the even one
        1.0 + 2.0 ** -8 + 2.0 ** -20: 0x3F81,    # just above halfway: up
        -2.5: 0xC020,
        0.0: 0x0000,
    }
    for v, bits in cases.items():
        assert int(inputs.to_bf16_bits(np.array([v], dtype=np.float32))[0]) == bits, v
    assert one == inputs.bf16_bits_to_f32(np.array([0x3F80], dtype=np.uint16))[0]
    x = np.random.default_rng(3).standard_normal(100000).astype(np.float32) * np.float32(37.0)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(inputs.to_bf16_bits(x), ref)
    # decoding is exact: bf16 values survive the round trip
    assert np.array_equal(inputs.to_bf16_bits(inputs.bf16_bits_to_f32(ref)), ref)


def test_requested_distributions():
    w = inputs.bf16_bits_to_f32(inputs.normal_bf16((400, 500), 0.02, 9)).astype(np.float64)
    assert abs(w.mean()) < 5 * 0.02 / math.sqrt(w.size)
    assert abs(w.std() / 0.02 - 1.0) < 0.01
    x = inputs.activations_f32(64, 4096).astype(np.float64)
    assert abs(x.std() - 1.0) < 0.01
    lut = inputs.routing_lut(200000, 0.3)
    assert abs(lut.mean() - 0.3) < 0.005
    V, s, n = 1000, 1.1, 200000
    ids = inputs.token_ids_zipf(n, V, s=s)
    assert ids.min() >= 0 and ids.max() < V
    p1 = 1.0 / sum(r ** -s for r in range(1, V + 1))       # rank 1 -> token id 0
    assert abs(np.mean(ids == 0) - p1) < 4 * math.sqrt(p1 * (1 - p1) / n)
    xc = inputs.bf16_bits_to_f32(inputs.activations_correlated_bf16(3, 20000, 0.9)).astype(np.float64)
    assert abs(np.corrcoef(xc[0], xc[1])[0, 1] - 0.81) < 0.02


def test_stack_sparsity_targets_are_the_stated_grid():
    L = 32
    t = inputs.stack_sparsity_targets(L, 0.55, 0.85)
    np.testing.assert_allclose(np.sort(t), 0.55 + 0.30 * (np.arange(L) + 0.5) / L, rtol=0, atol=1e-15)
    assert abs(t.mean() - 0.70) < 1e-12
    assert not np.array_equal(t, np.sort(t))   # assigned to the blocks by a seeded shuffle
