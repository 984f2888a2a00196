"""GPU routing calibration (Sec. 3.2, Eqs. 11-14) against the oracle: per-token
scores, the routing threshold chosen on a held-out split, and the table."""
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


@pytest.mark.parametrize("V,n,m", [(1000, 20000, 5000), (151936, 400000, 100000)])
def test_route_calibration_matches_oracle(sats, oracle, V, n, m):
    ids, lb, ls = inputs.routing_corpus(n, V)
    held = inputs.token_ids_zipf(m, V, seed=inputs.SEED_IDS + 200)
    score = sats.token_scores(P.dev(ids), P.dev(lb), P.dev(ls), V)
    s_ref = oracle.token_scores(ids, lb, ls, V)
    sg = score.cpu().numpy().astype(np.float64)
    assert np.array_equal(np.isinf(sg), np.isinf(s_ref))
    fin = np.isfinite(s_ref)
    np.testing.assert_allclose(sg[fin], s_ref[fin], rtol=1e-6, atol=1e-7)
    for r_tar in (0.25, 0.5, 0.75):
        tau, R, lut = sats.route_calibrate(score, P.dev(held), r_tar)
        # Eq. 14 on the library's own scores picks the same threshold
        tau_ref, R_ref = oracle.route_threshold(sg, held, r_tar)
        assert tau == tau_ref and R == R_ref
        assert np.array_equal(lut.cpu().numpy(), oracle.route_lut(sg, tau))
        assert abs(R - r_tar) < 0.05


def test_bad_token_id_is_reported(sats):
    ids = torch.tensor([0, 1, 7], dtype=torch.int32, device="cuda")
    lb = torch.zeros(3, device="cuda")
    with pytest.raises(sats.SatsError) as e:
        sats.token_scores(ids, lb, lb, 5)
    assert e.value.status == sats.EDEVICE
