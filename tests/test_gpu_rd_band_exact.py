"""The r_d band decision of Eq. 4, exact against float64.

Given log pi_old and log mu_old as float32 inputs, log r_d = log pi_old -
log mu_old involves no log-sum-exp, so the kernel's decision must equal the
float64 one for every token, however close to a band edge: the kernel forms
the difference and holds the thresholds in float-float (about 48 bits).  The
inputs put every token a few float32 steps from a band edge (about 1800 of
65536 within 1e-8 of it), where a float32 subtraction decides hundreds wrongly
(checked below, so that the test can see such a mistake).
"""

import numpy as np
import pytest
import torch

from paper_2605_12070_gb300 import occ

pytestmark = pytest.mark.gpu

RD_LO, RD_HI = 0.8, 1.25


def _inputs(T, seed):
    rng = np.random.default_rng(seed)
    lp_old = (-rng.uniform(1e-3, 6.0, T)).astype(np.float32)
    edge = np.where(rng.random(T) < 0.5, np.log(RD_LO), np.log(RD_HI))
    ideal = lp_old.astype(np.float64) - edge            # log mu_old on the edge
    lp_mu = ideal.astype(np.float32)
    k = rng.integers(-2, 3, T).astype(np.float32)       # a few float32 steps either side
    lp_mu = (lp_mu + k * np.spacing(np.abs(lp_mu))).astype(np.float32)
    return lp_old, lp_mu


@pytest.mark.parametrize("seed", [0, 1])
def test_rd_band_is_float64_exact_near_the_edges(seed):
    T, V = 65536, 64
    lp_old, lp_mu = _inputs(T, seed)
    log_rd = lp_old.astype(np.float64) - lp_mu.astype(np.float64)   # exact
    lo, hi = np.log(RD_LO), np.log(RD_HI)
    want = (log_rd >= lo) & (log_rd <= hi)
    dist = np.minimum(np.abs(log_rd - lo), np.abs(log_rd - hi))
    assert (dist < 1e-8).sum() > 1000          # the inputs sit on the edges
    f32 = (lp_old - lp_mu).astype(np.float64)  # a float32 subtraction decides some wrongly
    assert (((f32 >= lo) & (f32 <= hi)) != want).sum() > 0

    g = torch.Generator(device="cuda").manual_seed(seed)
    z = torch.randn((T, V), generator=g, device="cuda")
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    adv = torch.randn(T, generator=g, device="cuda")
    out = occ.occ_decoupled_loss_fwd_bwd(
        z, ids, torch.from_numpy(lp_old).cuda(), torch.from_numpy(lp_mu).cuda(), adv, None,
        rd_lo=RD_LO, rd_hi=RD_HI, eps_low=0.2, eps_high=0.28, dlogits=None)
    torch.cuda.synchronize()
    got = (out["flags"].cpu().numpy() & occ.FLAG_IN_BAND) != 0
    sharp = dist > 1e-13
    assert sharp.sum() > T - 50
    assert np.array_equal(got[sharp], want[sharp])
