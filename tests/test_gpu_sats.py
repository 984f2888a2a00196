"""GPU SATS calibration (Sec. 3.1, Eqs. 3, 6-10) against the oracle.

- sats_layer_err (Eq. 6) at thresholds that fall between two neurons' |a|
  (so that the GPU's fp32 gate values and the oracle's fp64 ones make the same
  mask decisions): errors and sparsities match;
- sats_sats_calibrate on a small stack, step by step: the coarse candidates
  are the oracle's Eq. 3 percentiles of its own dense-stack inputs; every
  error in the returned table matches the oracle's Eq. 6 at that threshold
  (for a candidate that is itself some neuron's |a|, between the oracle's
  values just below and just above it); the guardrail threshold is the
  oracle's percentile at the target; and the choice of b*, T*(b*) is the
  oracle's Eqs. 7-10 applied to the same table; the fine candidates are the
  oracle's (the same coarse choice, the same placement between its neighbours).
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


def _gap_thresholds(a, qs):
    """Thresholds halfway between consecutive distinct |a| order statistics near quantiles qs,
    at a gap of at least 1e-4 relative (no value within 5e-5 of the threshold)."""
    v = np.unique(np.abs(a).ravel())
    out = []
    for q in qs:
        i = int(q * (v.size - 1))
        while i + 1 < v.size and (v[i + 1] - v[i]) < 1e-4 * v[i + 1]:
            i += 1
        out.append(float(np.float32(0.5 * (v[i] + v[i + 1]))))
    return out


@pytest.mark.parametrize("C", [2, 16])
def test_layer_err_matches_oracle(sats, oracle, C):
    H, N = 256, 512
    w = inputs.mlp_weights(H, N, std=0.05, seed=70)
    x = inputs.activations_f32(C, H, seed=71)
    x64 = x.astype(np.float64)
    a = oracle.gate_act(x64, w.Wg)
    ts = [0.0] + _gap_thresholds(a, [0.1, 0.3, 0.5, 0.7, 0.9]) + [float(np.abs(a).max() * 2)]
    layer = sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd))
    err, sp = sats.layer_err(layer, P.dev(x), ts, eps=1e-6)
    e_ref, s_ref = oracle.layer_err(x64, w.Wg, w.Wu, w.Wd, ts, eps=1e-6)
    assert err[0] == 0.0 or abs(err[0]) < 1e-6        # t = 0 removes nothing
    np.testing.assert_allclose(err, e_ref, rtol=1e-3, atol=2e-5)
    np.testing.assert_allclose(sp, s_ref, rtol=0, atol=1e-12)
    layer.close()


def test_sats_calibrate_matches_oracle_step_by_step(sats, oracle):
    L, H, N, C = 3, 256, 512, 16
    K0, K1, s_tar, eps = 10, 4, 0.5, 1e-5
    ws_ = [inputs.mlp_weights(H, N, layer=l, std=0.05, seed=80) for l in range(L)]
    nw = [inputs.norm_weight(H, layer=l) for l in range(L)]
    x = inputs.activations_f32(C, H, seed=81)
    layers = [sats.Layer(P.dev_u16(w.Wg), P.dev_u16(w.Wu), P.dev_u16(w.Wd)) for w in ws_]
    r = sats.sats_calibrate(layers, [P.dev(v) for v in nw], eps, P.dev(x), s_tar, K0=K0, K1=K1, guardrail=True)
    tt, te, tsp = (np.asarray(m) for m in r["table"])
    Kc = K0 - 1
    assert tt.shape == (L, Kc + K1)

    # the oracle's dense stack and its Eq. 3 candidates
    xs = x.astype(np.float64)
    n_in = []
    for l in range(L):
        n = oracle.rmsnorm(xs, nw[l], eps)
        n_in.append(n)
        xs = xs + oracle.dense_mlp(n, ws_[l].Wg, ws_[l].Wu, ws_[l].Wd)
    for l in range(L):
        a = oracle.gate_act(n_in[l], ws_[l].Wg)
        cand = [oracle.percentile_threshold(a, k / K0) for k in range(1, K0)]
        np.testing.assert_allclose(tt[l, :Kc], cand, rtol=1e-4)
        # Eq. 6 at every threshold of the table
        lo, slo = oracle.layer_err(n_in[l], ws_[l].Wg, ws_[l].Wu, ws_[l].Wd, tt[l] * (1 - 1e-4))
        hi, shi = oracle.layer_err(n_in[l], ws_[l].Wg, ws_[l].Wu, ws_[l].Wd, tt[l] * (1 + 1e-4))
        assert np.all(te[l] >= np.minimum(lo, hi) * (1 - 2e-3) - 2e-5)
        assert np.all(te[l] <= np.maximum(lo, hi) * (1 + 2e-3) + 2e-5)
        assert np.all(tsp[l] >= np.minimum(slo, shi) - 1e-12) and np.all(tsp[l] <= np.maximum(slo, shi) + 1e-12)
    # guardrail: the last block keeps the CATS threshold at the target
    g_t = oracle.percentile_threshold(oracle.gate_act(n_in[L - 1], ws_[L - 1].Wg), s_tar)
    assert r["t"][L - 1] == pytest.approx(g_t, rel=1e-4)
    # Eqs. 7-10 on the returned table give the returned choice
    t_sel = np.asarray(r["t"], dtype=np.float64)
    sp_sel = [tsp[l][tt[l] == np.float32(t_sel[l])][0] if t_sel[l] > 0 else 0.0 for l in range(L - 1)]
    g_sp = r["S"] * L - sum(sp_sel)
    b2, t2, S2 = oracle.sats_select(tt, te, tsp, s_tar, L - 1, float(np.float32(r["t"][L - 1])), g_sp)
    assert b2 == r["b"]
    np.testing.assert_allclose(t2[:L - 1], t_sel[:L - 1], rtol=0, atol=0)
    assert abs(r["S"] - s_tar) < 0.1
    # the fine candidates (coarse-to-fine, step 5): the oracle's, placed between the coarse
    # neighbours of the same coarse choice, to the fp32 rounding of the candidates
    r_or = oracle.sats_calibrate(x.astype(np.float64), [w.Wg for w in ws_], [w.Wu for w in ws_],
                                 [w.Wd for w in ws_], nw, eps, s_tar, K0=K0, K1=K1, guardrail=True)
    np.testing.assert_allclose(tt[:, Kc:], r_or["fine"][0][:, Kc:], rtol=1e-4)
    for l in layers:
        l.close()
