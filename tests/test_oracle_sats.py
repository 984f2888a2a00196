"""Pins for the oracle's SATS calibration (Sec. 3.1, Eqs. 6-10; Sec. 4 guardrail).

Eq. 6 is pinned by its closed forms: nothing removed (t = 0) gives error 0,
everything removed gives 1 (eps = 0); a single neuron turns each token's error
into 0 or 1; with W_down the identity the error is the norm of the removed
part of h over the norm of h; scaling W_down changes nothing.  Eqs. 7-10 are
pinned by tables worked by hand, including a non-monotone error curve and the
final-block guardrail; the coarse-to-fine driver by what its steps guarantee.
"""
import numpy as np
import pytest

from paper_2607_08991_gb300 import inputs

BF16_ONE = 0x3F80
BF16_TWO = 0x4000


def _x(C, H, seed=3):
    return inputs.activations_f32(C, H, seed=seed).astype(np.float64)


# ---------------------------------------------------------------- Eq. 6

def test_err_nothing_and_everything_removed(oracle):
    H, N, C = 32, 48, 5
    w = inputs.mlp_weights(H, N, std=0.2)
    x = _x(C, H)
    a = oracle.gate_act(x, w.Wg)
    big = float(np.abs(a).max()) * 2.0
    err, sp = oracle.layer_err(x, w.Wg, w.Wu, w.Wd, [0.0, big], eps=0.0)
    assert err[0] == 0.0 and sp[0] == 0.0          # t = 0 keeps every neuron: y~ = y
    assert err[1] == pytest.approx(1.0, rel=1e-15)  # t > max|a| removes all: ||y|| / ||y||
    assert sp[1] == 1.0


def test_err_single_neuron_is_fraction_of_tokens_removed(oracle):
    H, N, C = 8, 1, 12
    w = inputs.mlp_weights(H, N, std=0.5)
    x = _x(C, H, seed=7)
    a = np.abs(oracle.gate_act(x, w.Wg)[:, 0])
    t = 0.5 * (np.sort(a)[5] + np.sort(a)[6])      # between two tokens' |a|, no tie
    err, sp = oracle.layer_err(x, w.Wg, w.Wu, w.Wd, [t], eps=0.0)
    removed = float(np.mean(a < t))
    assert removed == pytest.approx(6 / 12)
    assert err[0] == pytest.approx(removed, rel=1e-15)  # per token: 0 if kept, 1 if removed
    assert sp[0] == pytest.approx(removed, rel=1e-15)


def test_err_with_identity_down_projection(oracle):
    # W_down = I (N = H): y = h, so Err = mean_c ||h_c restricted to removed j|| / ||h_c||.
    H = N = 16
    C = 6
    w = inputs.mlp_weights(H, N, std=0.3, seed=21)
    Wd = np.zeros((N, H), np.uint16)
    np.fill_diagonal(Wd, BF16_ONE)
    x = _x(C, H, seed=9)
    a = oracle.gate_act(x, w.Wg)
    u = oracle.up_proj(x, w.Wu)
    h = a * u
    ts = np.quantile(np.abs(a), [0.2, 0.5, 0.8]) * (1.0 + 1e-9)
    err, sp = oracle.layer_err(x, w.Wg, w.Wu, Wd, ts, eps=0.0)
    for k, t in enumerate(ts):
        rem = np.abs(a) < t
        ref = np.mean(np.linalg.norm(np.where(rem, h, 0.0), axis=1) / np.linalg.norm(h, axis=1))
        assert err[k] == pytest.approx(ref, rel=1e-12)
        assert sp[k] == pytest.approx(rem.mean(), rel=1e-15)


def test_err_is_invariant_to_scaling_w_down(oracle):
    H, N, C = 24, 40, 4
    w = inputs.mlp_weights(H, N, std=0.2, seed=4)
    x = _x(C, H, seed=2)
    # multiply every W_down entry by 2 exactly: add one to the bf16 exponent
    Wd2 = w.Wd.copy()
    nz = (Wd2 & 0x7FFF) != 0
    Wd2[nz] = Wd2[nz] + 0x0080
    ts = [0.01, 0.03, 0.08]
    e1, s1 = oracle.layer_err(x, w.Wg, w.Wu, w.Wd, ts, eps=0.0)
    e2, s2 = oracle.layer_err(x, w.Wg, w.Wu, Wd2, ts, eps=0.0)
    np.testing.assert_allclose(e1, e2, rtol=1e-13)
    np.testing.assert_array_equal(s1, s2)


def test_sparsity_is_monotone_in_t(oracle):
    H, N, C = 32, 64, 6
    w = inputs.mlp_weights(H, N, std=0.2, seed=8)
    x = _x(C, H, seed=5)
    ts = np.linspace(0.0, 0.5, 21)
    _, sp = oracle.layer_err(x, w.Wg, w.Wu, w.Wd, ts)
    assert np.all(np.diff(sp) >= 0.0)


# ---------------------------------------------------------------- Eqs. 7-10

# Two blocks, three candidates each (worked by hand):
#   budget b : T*(b)        S(b)
#   0        : (0,   0  )   0
#   0.01     : (0.1, 0  )   (0.3 + 0  ) / 2 = 0.15
#   0.02     : (0.1, 0.1)   (0.3 + 0.2) / 2 = 0.25
#   0.03     : (0.1, 0.2)   (0.3 + 0.6) / 2 = 0.45
#   0.05     : (0.2, 0.2)   (0.5 + 0.6) / 2 = 0.55
#   0.1      : (0.2, 0.3)   (0.5 + 0.8) / 2 = 0.65
#   0.2      : (0.3, 0.3)   (0.7 + 0.8) / 2 = 0.75
T = np.array([[0.1, 0.2, 0.3], [0.1, 0.2, 0.3]])
ERR = np.array([[0.01, 0.05, 0.2], [0.02, 0.03, 0.1]])
SP = np.array([[0.3, 0.5, 0.7], [0.2, 0.6, 0.8]])


@pytest.mark.parametrize("s_tar,b,t,S", [
    (0.52, 0.05, [0.2, 0.2], 0.55),
    (0.44, 0.03, [0.1, 0.2], 0.45),
    (0.71, 0.2, [0.3, 0.3], 0.75),
    (0.10, 0.01, [0.1, 0.0], 0.15),
    (0.02, 0.0, [0.0, 0.0], 0.0),
])
def test_select_worked_table(oracle, s_tar, b, t, S):
    bb, tt, SS = oracle.sats_select(T, ERR, SP, s_tar)
    assert bb == b
    np.testing.assert_array_equal(tt, t)
    assert SS == pytest.approx(S, abs=1e-15)


def test_select_takes_the_largest_admissible_threshold(oracle):
    # Eq. 7 is a max over thresholds, not over the error curve: with a
    # non-monotone error the larger threshold is admissible at a smaller budget.
    t = np.array([[0.1, 0.2]])
    err = np.array([[0.3, 0.1]])
    sp = np.array([[0.4, 0.6]])
    b, tt, S = oracle.sats_select(t, err, sp, 0.6)
    assert b == 0.1 and tt[0] == 0.2 and S == pytest.approx(0.6)
    b, tt, S = oracle.sats_select(t, err, sp, 0.45)      # 0.4 needs b = 0.3, where t* = 0.2 again
    assert tt[0] == 0.2


def test_select_guardrail_block(oracle):
    # block 1 fixed at t = 0.25 with sparsity 0.7; block 0 chosen so the mean approaches s_tar
    b, tt, S = oracle.sats_select(T, ERR, SP, 0.5, guard=1, guard_t=0.25, guard_sp=0.7)
    # candidates for block 0 give S = (sp0 + 0.7) / 2: 0.35 (t=0), 0.5 (0.1), 0.6 (0.2), 0.7 (0.3)
    assert tt[1] == 0.25 and tt[0] == 0.1 and S == pytest.approx(0.5) and b == 0.01


def test_select_result_is_closest_over_all_budgets(oracle):
    rng = np.random.default_rng(5)
    for _ in range(20):
        L, K = 3, 5
        t = np.sort(rng.random((L, K)), axis=1)
        sp = np.sort(rng.random((L, K)), axis=1)
        err = rng.random((L, K)) * 0.1
        s_tar = float(rng.random())
        b, tt, S = oracle.sats_select(t, err, sp, s_tar)
        # the chosen thresholds are admissible at b, and none larger is
        for l in range(L):
            adm = t[l][err[l] <= b]
            assert tt[l] == (adm.max() if adm.size else 0.0)
        # no other budget comes closer to the target
        for bb in np.concatenate([[0.0], err.ravel()]):
            S2 = np.mean([sp[l][t[l] == (t[l][err[l] <= bb].max())][0] if (err[l] <= bb).any() else 0.0
                          for l in range(L)])
            assert abs(S - s_tar) <= abs(S2 - s_tar) + 1e-15


# ---------------------------------------------------------------- coarse-to-fine driver

def _stack(L, H, N, seed=30):
    ws = [inputs.mlp_weights(H, N, layer=l, std=0.05, seed=seed) for l in range(L)]
    nw = [inputs.norm_weight(H, layer=l) for l in range(L)]
    return ws, nw


@pytest.mark.slow
def test_calibrate_hits_the_target_within_the_candidate_spacing(oracle):
    L, H, N, C = 3, 32, 64, 6
    ws, nw = _stack(L, H, N)
    x = _x(C, H, seed=11)
    r = oracle.sats_calibrate(x, [w.Wg for w in ws], [w.Wu for w in ws], [w.Wd for w in ws], nw, 1e-5, 0.5,
                              K0=10, K1=6, guardrail=True)
    t_all, e_all, s_all = r["fine"]
    # the guardrail block keeps the Eq. 3 percentile at the target
    n_last = x.copy()
    for l in range(L - 1):
        n = oracle.rmsnorm(n_last, nw[l], 1e-5)
        n_last = n_last + oracle.dense_mlp(n, ws[l].Wg, ws[l].Wu, ws[l].Wd)
    n = oracle.rmsnorm(n_last, nw[L - 1], 1e-5)
    assert r["t"][L - 1] == oracle.percentile_threshold(oracle.gate_act(n, ws[L - 1].Wg), 0.5)
    # every other block's threshold is a candidate admissible at b*, and the largest one
    for l in range(L - 1):
        adm = t_all[l][e_all[l] <= r["b"]]
        assert r["t"][l] == (adm.max() if adm.size else 0.0)
    # the coarse candidates are increasing percentiles (their fine neighbours are pinned below)
    coarse_t = r["coarse"][0]
    assert np.all(np.diff(coarse_t, axis=1) >= 0.0)
    assert abs(r["S"] - 0.5) < 0.1


# ---------------------------------------------------------------- coarse-to-fine: the fine candidates
#
# A one-block stack worked by hand (H = 1, N = 2, two calibration tokens, RMSNorm with eps = 0 and
# gain 1, so the block inputs are n = +1 and n = -1; W_gate = [1, 2], W_up = [1, 1],
# W_down = [1, 1]^T, so y = n * sum_j keep_j a_j).  The four post-gate magnitudes are
#   |SiLU(-2)| = 2 / (1 + e^2),  |SiLU(-1)| = 1 / (1 + e),  SiLU(1) = 1 / (1 + e^-1),  SiLU(2) = 2 / (1 + e^-2)
# in increasing order.  With K0 = 4 the coarse candidates are the Eq. 3 percentiles at 1/4, 2/4, 3/4:
# the first three magnitudes (m = ceil(k n) = k of n = 4 values).  Eq. 6 at each (token 0 keeps both
# neurons below SiLU(1); token 1 loses |SiLU(-2)| at the second and both at the third):
#   t1: err 0,                                        sp 0
#   t2: err (0 + |SiLU(-2)| / (|SiLU(-1)| + |SiLU(-2)|)) / 2,  sp 1/4
#   t3: err (0 + 1) / 2,                              sp 1/2
# Eqs. 7-10 then pick t2 for s_tar = 0.3, t3 for 0.45 and t1 for 0, and step 5 places K1 = 3
# candidates at lo + (hi - lo) k / 4 between the coarse neighbours of that choice: (t1, t3), (t2, max|a|)
# and (0, t2) respectively.

def _silu(z):
    import math
    return z / (1.0 + math.exp(-z))


def _worked_block():
    bits = lambda v: (np.asarray(v, np.float32).view(np.uint32) >> 16).astype(np.uint16)
    Wg = bits([[1.0, 2.0]])
    Wu = bits([[1.0, 1.0]])
    Wd = bits([[1.0], [1.0]])
    x = np.array([[1.0], [-1.0]])
    return x, Wg, Wu, Wd, [np.ones(1, np.float32)]


@pytest.mark.parametrize("s_tar,lo,hi", [
    (0.3, lambda m: m[0], lambda m: m[2]),
    (0.45, lambda m: m[1], lambda m: m[3]),
    (0.0, lambda m: 0.0, lambda m: m[1]),
])
def test_fine_candidates_of_a_worked_block(oracle, s_tar, lo, hi):
    x, Wg, Wu, Wd, nw = _worked_block()
    mags = [abs(_silu(-2.0)), abs(_silu(-1.0)), _silu(1.0), _silu(2.0)]   # increasing
    r = oracle.sats_calibrate(x, [Wg], [Wu], [Wd], nw, 0.0, s_tar, K0=4, K1=3, guardrail=False, err_eps=0.0)
    cand, err0, sp0 = r["coarse"]
    np.testing.assert_allclose(cand[0], mags[:3], rtol=1e-14)
    e2 = 0.5 * mags[0] / (mags[0] + mags[1])
    np.testing.assert_allclose(err0[0], [0.0, e2, 0.5], rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(sp0[0], [0.0, 0.25, 0.5], rtol=0, atol=0)
    fine = r["fine"][0][0, 3:]
    expect = [lo(mags) + (hi(mags) - lo(mags)) * k / 4.0 for k in (1, 2, 3)]
    np.testing.assert_allclose(fine, expect, rtol=1e-13)


def test_final_choice_can_be_a_fine_candidate(oracle):
    # s_tar = 0.7: the coarse S(b) takes 0, 1/4 and 1/2, so the coarse choice is t3 = SiLU(1) and the
    # fine candidates lie between t2 and SiLU(2):
    #   f1 = t2 + (SiLU(2) - t2) / 4  (below SiLU(1): token 0 keeps both, token 1 none: err 1/2, sp 1/2)
    #   f2, f3 above SiLU(1): token 0 also loses SiLU(1): err (SiLU(1) / (SiLU(1) + SiLU(2)) + 1) / 2, sp 3/4
    # Over coarse and fine candidates S(b) takes 0, 1/4, 1/2 (at b = 1/2, t*(1/2) = t3, which is
    # larger than f1) and 3/4 (at b = that error: t* = f3, the largest admissible); 3/4 is the
    # closest to 0.7, so the block takes f3.  At s_tar = 0.45 the same table gives 1/2 and t3.
    x, Wg, Wu, Wd, nw = _worked_block()
    m = [abs(_silu(-2.0)), abs(_silu(-1.0)), _silu(1.0), _silu(2.0)]
    r = oracle.sats_calibrate(x, [Wg], [Wu], [Wd], nw, 0.0, 0.7, K0=4, K1=3, guardrail=False, err_eps=0.0)
    f3 = m[1] + (m[3] - m[1]) * 3.0 / 4.0
    e_hi = 0.5 * (m[2] / (m[2] + m[3]) + 1.0)
    t_all, e_all, s_all = r["fine"]
    np.testing.assert_allclose(e_all[0, 3:], [0.5, e_hi, e_hi], rtol=1e-12)
    np.testing.assert_allclose(s_all[0, 3:], [0.5, 0.75, 0.75], rtol=0, atol=0)
    assert r["t"][0] == pytest.approx(f3, rel=1e-13)
    assert r["b"] == pytest.approx(e_hi, rel=1e-12) and r["S"] == 0.75
    r = oracle.sats_calibrate(x, [Wg], [Wu], [Wd], nw, 0.0, 0.45, K0=4, K1=3, guardrail=False, err_eps=0.0)
    assert r["t"][0] == pytest.approx(m[2], rel=1e-13) and r["S"] == 0.5


@pytest.mark.slow
@pytest.mark.parametrize("s_tar", [0.5, 0.97])
def test_fine_candidates_sit_evenly_between_the_coarse_neighbours(oracle, s_tar):
    # on a random 3-block stack: for every block but the guardrail block, the K1 fine candidates are
    # evenly spaced and strictly inside (lower, upper), where lower is the largest coarse candidate
    # below the coarse choice t*_l (0 if none) and upper the smallest above it (else the block's
    # largest |a| on its dense-stack inputs).  At s_tar = 0.97, above every coarse sparsity, each
    # block's coarse choice is its largest candidate, so upper is that block's own largest |a|.
    L, H, N, C, K0, K1 = 3, 32, 64, 6, 10, 6
    ws, nw = _stack(L, H, N)
    x = _x(C, H, seed=11)
    r = oracle.sats_calibrate(x, [w.Wg for w in ws], [w.Wu for w in ws], [w.Wd for w in ws], nw, 1e-5, s_tar,
                              K0=K0, K1=K1, guardrail=True)
    cand, err0, sp0 = r["coarse"]
    g_t, g_sp = r["guard"]
    _, t0, _ = oracle.sats_select(cand, err0, sp0, s_tar, L - 1, g_t, g_sp)
    if s_tar > 0.9:
        assert np.all(t0[:L - 1] == cand[:L - 1, -1])
    fine = r["fine"][0][:, K0 - 1:]
    xs = x.copy()
    for l in range(L):
        n = oracle.rmsnorm(xs, nw[l], 1e-5)
        amax = float(np.abs(oracle.gate_act(n, ws[l].Wg)).max())
        xs = xs + oracle.dense_mlp(n, ws[l].Wg, ws[l].Wu, ws[l].Wd)
        if l == L - 1:
            continue
        below = cand[l][cand[l] < t0[l]]
        above = cand[l][cand[l] > t0[l]]
        lower = below.max() if below.size else 0.0
        upper = above.min() if above.size else amax
        f = fine[l]
        assert np.all(f > lower) and np.all(f < upper)
        step = (upper - lower) / (K1 + 1)
        np.testing.assert_allclose(np.diff(np.concatenate([[lower], f, [upper]])), step, rtol=1e-9)
