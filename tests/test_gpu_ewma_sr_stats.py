"""Statistical pins of the bf16 proximal buffer's stochastic rounding, on the
kernel's own output.

The bit-exact tests of the bf16 EWMA compare the kernel with the oracle's
model of the same rounding; these tests instead check what stochastic
rounding is for, against quantities that do not depend on how the random bits
are laid out:

  * one step is unbiased: each stored bf16 value is one of the two bf16
    neighbours of the exact update v = tp + b (theta - tp) (App. B), and the
    mean of (stored - v), in bf16 units in the last place, is zero within a
    99.99 % confidence bound (the error of one rounding lies in (-1, 1) ulp and
    has standard deviation <= 1/2 ulp);
  * over 300 steps at beta = 0.99 the buffer tracks the float64 App. B
    recursion on the same parameter sequence: the mean error over the buffer
    stays within a bound derived from the recursion, sqrt(1 / (4 (1 - a^2)))
    ulp per element for the stationary error, divided by sqrt(n).  Nearest
    rounding, whose steps here are below half an ulp, freezes the buffer and
    misses the same bound by orders of magnitude.

Parameters live in [1, 2), where the bf16 unit in the last place is 2^-7 for
every element, so errors average in one unit.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2605_12070_gb300 import occ

pytestmark = pytest.mark.gpu

ULP = 2.0 ** -7     # bf16 spacing in [1, 2)
BETA = 0.99
Z = 4.0             # 99.99 % two-sided normal quantile (3.89), rounded up


def _start(n, seed):
    rng = np.random.default_rng(seed)
    th0 = (1.5 + rng.uniform(-0.2, 0.2, n)).astype(np.float32)
    tp0 = torch.from_numpy(th0).to(torch.bfloat16)   # nearest-rounded start
    return th0, tp0


def _bf16_f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def test_one_step_is_unbiased_against_the_exact_update():
    n = 1 << 24
    th0, tp0 = _start(n, 1)
    # a step of about 0.3 ulp toward theta for every element: nearest rounding
    # would keep every value and err by -0.3 ulp on average
    rng = np.random.default_rng(2)
    th = (_bf16_f64(tp0) + rng.uniform(20, 40, n) * ULP).astype(np.float32)
    tp = tp0.to("cuda")
    st = occ.new_ewma_state("cuda", w0=1.0 / (1.0 - BETA))
    occ.occ_ewma_update_bf16(tp, torch.from_numpy(th).cuda(), BETA, st, sr_seed=12345)
    torch.cuda.synchronize()
    s = occ.decode_ewma_state(st)
    assert s.coef_b == pytest.approx(1.0 - BETA, abs=1e-15)
    before = _bf16_f64(tp0)
    v = before + s.coef_b * (th.astype(np.float64) - before)     # App. B, float64
    got = _bf16_f64(tp)
    lo = np.floor(v / ULP) * ULP
    assert np.all((got == lo) | (got == lo + ULP)), "a value is not a bf16 neighbour of v"
    err = (got - v) / ULP
    bound = Z * 0.5 / np.sqrt(n) + 2.0 ** -14   # + the float32 rounding of v
    assert abs(err.mean()) <= bound, (err.mean(), bound)
    # the fraction of values rounded up matches the fractional parts
    frac = (v - lo) / ULP
    up = got > lo
    z = (up.sum() - frac.sum()) / np.sqrt(np.sum(frac * (1 - frac)))
    assert abs(z) <= Z + 0.5, z


@pytest.mark.parametrize("mode", ["stochastic", "nearest"])
def test_300_steps_track_the_float64_recursion(mode):
    n, steps = 1 << 20, 300
    th0, tp0 = _start(n, 3)
    drift = np.float32(0.02 * ULP)       # theta moves 0.02 ulp per step
    tp = tp0.to("cuda")
    st = occ.new_ewma_state("cuda", w0=1.0 / (1.0 - BETA))
    ref = _bf16_f64(tp0)
    ost = oracle.EwmaState(w=1.0 / (1.0 - BETA))
    # stationary error of the recursion e' = a e + u, |u| < 1 ulp with
    # sd <= 1/2: per element sd <= sqrt(1 / (4 (1 - a^2))) ulp
    sd_elem = np.sqrt(1.0 / (4.0 * (1.0 - BETA ** 2)))
    bound = Z * sd_elem / np.sqrt(n) + 0.005   # + accumulated float32 roundings
    worst = 0.0
    for k in range(1, steps + 1):
        th = (th0 + np.float32(k) * drift).astype(np.float32)
        occ.occ_ewma_update_bf16(tp, torch.from_numpy(th).cuda(), BETA, st,
                                 sr_seed=(1000 + k) if mode == "stochastic" else 0)
        ref, ost, _ = oracle.ewma_update(ref, th, BETA, ost)
        if k % 50 == 0:
            torch.cuda.synchronize()
            mean_err = float(((_bf16_f64(tp) - ref) / ULP).mean())
            worst = max(worst, abs(mean_err))
    if mode == "stochastic":
        assert worst <= bound, (worst, bound)
    else:
        # the update steps (about 0.02 ulp) are below half an ulp: nearest
        # rounding keeps the buffer still while the recursion moves on
        assert worst > 100 * bound, (worst, bound)
