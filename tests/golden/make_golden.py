"""Writes the stored expected values under tests/golden/ (run: python tests/golden/make_golden.py).

Every value comes from the oracle (``oracle/``) on seeded inputs from
``paper_2607_08991_gb300.inputs``; nothing here computes the method itself.
The paper prints no worked example, so these files are regression fixtures:
they pin the oracle against accidental change, while the oracle's independent
pins (closed forms, brute force, invariants) live in tests/test_oracle_*.py.
"""
import os
import sys

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from paper_2607_08991_gb300 import inputs  # noqa: E402

H, N, B, C, K = 16, 24, 2, 4, 0.5
SEED = 31


def case():
    """The seeded inputs of the fixture: bf16 weights and activations, C calibration vectors."""
    w = inputs.mlp_weights(H, N, std=0.25, seed=SEED)
    xb = inputs.activations_bf16(B, H, seed=SEED + 1)
    cal = inputs.activations_bf16(C, H, seed=SEED + 2)
    return w, xb, cal


def main():
    oracle.build()
    w, xb, cal = case()
    t = oracle.percentile_threshold(oracle.gate_act(oracle.bf16_to_f64(cal), w.Wg), K)
    y, a, keep, _ = oracle.sparse_mlp(oracle.bf16_to_f64(xb), w.Wg, w.Wu, w.Wd, t)
    path = os.path.join(HERE, "sparse_mlp_h16_n24_b2.txt")
    with open(path, "w") as f:
        f.write("# Thresholded gated MLP (Sec. 2, Eqs. 1-5) at the 50th percentile threshold of the\n")
        f.write("# calibration activations (Eq. 3), H = %d, N = %d, B = %d tokens, %d calibration vectors;\n" % (H, N, B, C))
        f.write("# inputs: paper_2607_08991_gb300.inputs (weights std 0.25, seeds %d / %d / %d);\n" % (SEED, SEED + 1, SEED + 2))
        f.write("# values written by tests/golden/make_golden.py from the oracle only.\n")
        f.write("t %.17g\n" % t)
        for b in range(B):
            f.write("a%d %s\n" % (b, " ".join("%.17g" % v for v in a[b])))
            f.write("keep%d %s\n" % (b, "".join("1" if k else "0" for k in keep[b])))
            f.write("y%d %s\n" % (b, " ".join("%.17g" % v for v in y[b])))
    print(path)


if __name__ == "__main__":
    main()
