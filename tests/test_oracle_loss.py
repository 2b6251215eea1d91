"""Pins for the oracle's R2..R9 (ratios, band mask, PPO clip, token mean, gradient).

What fixes each expectation:
  * the decomposition r = r_d r_s of Eq. 1, checked against a brute-force
    softmax (math.fsum), which pins the direction of each log-ratio;
  * the special cases of Table 1: pi_theta = pi_old (r_s = 1, nothing clipped)
    and pi_old = mu_old (r_d = 1: standard PPO-clip & train_infer);
  * hand-built tokens on either side of every threshold for both advantage
    signs, with the outcome read off Eqs. 2-4;
  * the effective thresholds printed in Table 4 (tests/golden), reproduced by
    scanning the oracle's mask and clip decisions under the two interpolation
    proxies of App. A;
  * central finite differences of the oracle's loss (R6/R7) against its
    analytic gradient (R8), and torch autograd of the Eq. 2 surrogate;
  * counter recounts and the softmax-gradient invariant sum_v dz = 0.
"""

import math
import os

import numpy as np
import pytest

from oracle import (LossParams, decoupled_loss, proxy_logprob, token_logprob, token_terms,
                    FLAG_ACTIVE, FLAG_CLIPPED, FLAG_IN_BAND, FLAG_VALID)

P = LossParams(rd_lo=0.5, rd_hi=2.0, eps_low=0.2, eps_high=0.28)


def _tiny_batch(rng, T=6, V=9, old_noise=0.3, mu_noise=0.3):
    z = rng.normal(0, 2, size=(T, V))
    z_old = z + rng.normal(0, old_noise, size=(T, V))
    ids = rng.integers(0, V, size=T)
    lp_old, _ = token_logprob(z_old, ids)
    lp_mu = lp_old + rng.normal(0, mu_noise, size=T)
    adv = rng.normal(0, 1, size=T)
    return z, ids, lp_old, lp_mu, adv


def test_ratio_decomposition_against_brute_force():
    # Eq. 1: r_d r_s = pi_theta / mu_old with pi_theta from a brute-force softmax.
    rng = np.random.default_rng(10)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng)
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, None, P, want_dlogits=False)
    for t in range(len(ids)):
        den = math.fsum(math.exp(v) for v in z[t])
        pi_theta = math.exp(z[t, ids[t]]) / den
        r_total = pi_theta / math.exp(lp_mu[t])
        assert abs(out["r_d"][t] * out["r_s"][t] / r_total - 1) < 1e-12
        assert abs(out["r_s"][t] * math.exp(lp_old[t]) / pi_theta - 1) < 1e-12


def test_equal_policies_nothing_clipped():
    # pi_theta = pi_old: r_s = 1 exactly, MIS_ppo = 1 for both signs, and the
    # loss is -sum(m M_d w_d A) / N (Eq. 2 with r = 1).
    rng = np.random.default_rng(11)
    T, V = 40, 33
    z = rng.normal(0, 2, size=(T, V))
    ids = rng.integers(0, V, size=T)
    lp_old, _ = token_logprob(z, ids)
    lp_mu = lp_old + rng.normal(0, 0.5, size=T)   # some tokens leave the band
    adv = rng.normal(0, 1, size=T)
    mask = rng.random(T) < 0.8
    for rdw in (0, 1):
        p = LossParams(0.7, 1.4, 0.2, 0.28, rd_weight=rdw)
        out = decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, p)
        assert np.all(out["r_s"] == 1.0)
        assert out["n_clipped"] == 0
        N = int(mask.sum())
        acc = []
        for t in range(T):
            r_d = math.exp(lp_old[t] - lp_mu[t])
            if mask[t] and 0.7 <= r_d <= 1.4:
                acc.append(-(r_d if rdw else 1.0) * adv[t])
        assert abs(out["loss"] - math.fsum(acc) / N) < 1e-13
        assert 0 < out["n_rd_out"] < N


def test_old_equals_mu_reduces_to_standard_ppo():
    # Table 1, "PPO-clip & train_infer": r_d = 1 is always in band and the loss
    # is the plain Eq. 2 surrogate on r = pi_theta / mu_old.
    rng = np.random.default_rng(12)
    z, ids, lp_old, _, adv = _tiny_batch(rng, T=30)
    out = decoupled_loss(z, ids, lp_old, lp_old, adv, None, P)
    assert np.all(out["in_band"]) and out["n_rd_out"] == 0
    acc = []
    for t in range(30):
        den = math.fsum(math.exp(v) for v in z[t])
        r = math.exp(z[t, ids[t]]) / den / math.exp(lp_old[t])
        acc.append(min(r * adv[t], min(max(r, 0.8), 1.28) * adv[t]))
    assert abs(out["loss"] + math.fsum(acc) / 30) < 1e-13


# (advantage, r_s, expected clipped, expected surrogate s_t) read from Eqs. 2-3
# with eps_low = 0.2, eps_high = 0.28.
CLIP_CASES = [
    (+1.0, 1.50, True, 1.28),      # A >= 0 and r_s above 1+eps_high: clipped
    (+1.0, 1.28 * (1 - 1e-12), False, 1.28 * (1 - 1e-12)),  # just inside
    (+1.0, 1.28 * (1 + 1e-12), True, 1.28),                  # just outside
    (+1.0, 0.50, False, 0.50),     # A >= 0 never clips from below
    (-1.0, 0.50, True, -0.80),     # A < 0 and r_s below 1-eps_low: clipped
    (-1.0, 0.80 * (1 + 1e-12), False, -0.80 * (1 + 1e-12)),
    (-1.0, 0.80 * (1 - 1e-12), True, -0.80),
    (-1.0, 1.50, False, -1.50),    # A < 0 never clips from above
    (0.0, 3.00, True, 0.0),        # A = 0 takes the A >= 0 branch: clipped, s = 0
    (0.0, 0.10, False, 0.0),       # ... and is kept below 1+eps_high, s = 0
]


@pytest.mark.parametrize("A,r_s,clipped,s", CLIP_CASES)
def test_sign_dependent_clip_cases(A, r_s, clipped, s):
    lp_old = np.array([-2.0])
    lp_theta = lp_old + math.log(r_s)
    out = token_terms(lp_theta, lp_old, lp_old, np.array([A]), None, P)
    assert bool(out["flags"][0] & FLAG_CLIPPED) == clipped
    assert bool(out["flags"][0] & FLAG_ACTIVE) == (not clipped)
    assert abs(-out["loss_t"][0] - s) < 1e-12
    assert (out["g"][0] != 0.0) == (not clipped and A != 0.0)


@pytest.mark.parametrize("r_d,inside", [
    (0.5 * (1 + 1e-12), True), (0.5 * (1 - 1e-12), False),
    (2.0 * (1 - 1e-12), True), (2.0 * (1 + 1e-12), False), (1.0, True)])
def test_band_is_inclusive(r_d, inside):
    # M_[1/c,c](r) = 1{1/c <= r <= c} (Eq. 4): both ends belong to the band.
    lp_mu = np.array([-3.0])
    lp_old = lp_mu + math.log(r_d)
    out = token_terms(lp_old, lp_old, lp_mu, np.array([0.7]), None, P)
    assert bool(out["flags"][0] & FLAG_IN_BAND) == inside
    assert (out["loss_t"][0] != 0.0) == inside
    assert out["n_rd_out"] == (0 if inside else 1)


def _table4_rows(golden_dir):
    rows = []
    with open(os.path.join(golden_dir, "table4_effective_thresholds.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                v = line.split()
                rows.append((*map(float, v[:4]), int(v[4]), v[5], *map(float, v[6:])))
    return rows


def test_table4_effective_thresholds(golden_dir):
    """App. A / Table 4: with an interpolated proxy in place of pi_old, the
    oracle's mask and clip decisions cut the total ratio r_theta = pi_theta /
    mu_old exactly at the printed effective bounds (4 decimals)."""
    rows = _table4_rows(golden_dir)
    assert len(rows) == 24
    r_theta = np.linspace(0.95, 1.05, 200001)           # step 5e-7
    lp_mu = np.full(r_theta.size, -1.7)
    lp_theta = lp_mu + np.log(r_theta)
    for (mlo, mhi, clo, chi, n, kind, e_mlo, e_mhi, e_clo, e_chi) in rows:
        alpha = 1.0 / (n + 1)
        # Table 4's "Linear" rows are the arithmetic proxy (linear_prox of Table 1)
        lp_prox = proxy_logprob({"linear": "arithmetic"}.get(kind, kind), alpha, lp_mu, lp_theta)
        p = LossParams(mlo, mhi, 1.0 - clo, chi - 1.0)
        for A, which in ((1.0, "hi"), (-1.0, "lo")):
            out = token_terms(lp_theta, lp_prox, lp_mu, np.full(r_theta.size, A), None, p)
            band = r_theta[out["in_band"]]
            assert abs(band.min() - e_mlo) <= 5e-5 + 1e-6
            assert abs(band.max() - e_mhi) <= 5e-5 + 1e-6
            kept = r_theta[out["mis"]]
            if which == "hi":   # A >= 0 keeps r_theta below the effective upper clip
                assert kept.min() == r_theta[0]
                assert abs(kept.max() - e_chi) <= 5e-5 + 1e-6
            else:               # A < 0 keeps r_theta above the effective lower clip
                assert kept.max() == r_theta[-1]
                assert abs(kept.min() - e_clo) <= 5e-5 + 1e-6


def _loss_of(z, ids, lp_old, lp_mu, adv, mask, p):
    return decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, p, want_dlogits=False)["loss"]


@pytest.mark.parametrize("rdw", [0, 1])
def test_gradient_matches_central_differences(rdw):
    """R8 against central differences of R6/R7, h = 1e-6, on tokens at least
    1e-3 (log space) from every threshold, so no difference straddles a kink."""
    rng = np.random.default_rng(20 + rdw)
    T, V = 4, 16
    p = LossParams(0.8, 1.25, 0.2, 0.28, rd_weight=rdw, grad_scale=1.7)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=T, V=V, old_noise=0.4, mu_noise=0.15)
    mask = np.array([1, 1, 0, 1])
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, p)
    assert np.all(np.minimum(out["dist_rd"], out["dist_rs"]) > 1e-3)
    h = 1e-6
    fd = np.zeros((T, V))
    for t in range(T):
        for v in range(V):
            zp = z.copy(); zp[t, v] += h
            zm = z.copy(); zm[t, v] -= h
            fd[t, v] = (_loss_of(zp, ids, lp_old, lp_mu, adv, mask, p)
                        - _loss_of(zm, ids, lp_old, lp_mu, adv, mask, p)) / (2 * h)
    # d(loss)/dz is grad_scale-free; the oracle's dlogits carry grad_scale.
    np.testing.assert_allclose(out["dlogits"], p.grad_scale * fd, rtol=0, atol=1e-8)
    assert np.abs(fd).max() > 1e-3


def test_gradient_matches_autograd_of_eq2_surrogate():
    """R8 against torch autograd of the Eq. 2 surrogate with the Eq. 4 band
    mask, r_d held constant (it does not depend on theta)."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(30)
    T, V = 64, 11
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=T, V=V, old_noise=0.5, mu_noise=0.2)
    mask = rng.random(T) < 0.9
    for rdw in (0, 1):
        p = LossParams(0.75, 1.3, 0.2, 0.28, rd_weight=rdw)
        out = decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, p)
        zt = torch.tensor(z, dtype=torch.float64, requires_grad=True)
        lp = torch.log_softmax(zt, dim=1)[torch.arange(T), torch.tensor(ids)]
        r_s = torch.exp(lp - torch.tensor(lp_old))
        r_d = torch.exp(torch.tensor(lp_old - lp_mu))
        A = torch.tensor(adv)
        surr = torch.minimum(r_s * A, torch.clamp(r_s, 0.8, 1.28) * A)
        keep = torch.tensor(mask) & (r_d >= 0.75) & (r_d <= 1.3)
        w = r_d if rdw else torch.ones(T, dtype=torch.float64)
        objective = torch.where(keep, w * surr, torch.zeros_like(surr)).sum() / int(mask.sum())
        (-objective).backward()
        np.testing.assert_allclose(out["dlogits"], zt.grad.numpy(), rtol=0, atol=1e-14)
        assert abs(out["loss"] + objective.item()) < 1e-14


def test_softmax_gradient_rows_sum_to_zero_and_zero_rows():
    rng = np.random.default_rng(40)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=200, V=13, old_noise=0.6, mu_noise=0.5)
    adv[:10] = 0.0
    mask = rng.random(200) < 0.7
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, P)
    dz = out["dlogits"]
    np.testing.assert_allclose(dz.sum(axis=1), 0.0, atol=1e-15)
    dead = ~(out["flags"] & FLAG_ACTIVE).astype(bool) | (adv == 0.0)
    assert np.all(dz[dead] == 0.0)
    assert np.all(dz[:10] == 0.0)
    live = ~dead
    assert live.sum() > 50
    # the sampled token's entry is g (1 - p_y): same sign as g
    assert np.all(np.sign(dz[live, ids[live]]) == np.sign(out["g"][live]))


def test_counters_recount_from_flags():
    rng = np.random.default_rng(50)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=500, V=7, old_noise=0.7, mu_noise=0.6)
    mask = rng.random(500) < 0.85
    ids[3] = 7       # out of range: dropped and reported
    ids[4] = -2
    mask[3] = mask[4] = True
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, mask, P)
    n_valid = n_out = n_clip = n_act = 0
    for t in range(500):
        f = int(out["flags"][t])
        if f & FLAG_VALID:
            n_valid += 1
            n_out += not (f & FLAG_IN_BAND)
            n_clip += bool(f & FLAG_CLIPPED)
            n_act += bool(f & FLAG_ACTIVE)
            assert bool(f & FLAG_ACTIVE) == (bool(f & FLAG_IN_BAND) and not (f & FLAG_CLIPPED))
        else:
            assert f == 0
    assert (n_valid, n_out, n_clip, n_act) == (out["n_valid"], out["n_rd_out"],
                                               out["n_clipped"], out["n_active"])
    assert out["n_active"] <= out["n_valid"] - out["n_rd_out"]
    assert out["bad_ids"] == 2 and out["N"] == int(mask.sum()) - 2
    assert 0 < out["n_rd_out"] and 0 < out["n_clipped"]


def test_empty_and_all_masked():
    p = P
    out = decoupled_loss(np.zeros((0, 5)), np.zeros(0, dtype=int), np.zeros(0), np.zeros(0),
                         np.zeros(0), None, p)
    assert out["loss"] == 0.0 and out["N"] == 0 and out["dlogits"].shape == (0, 5)
    rng = np.random.default_rng(60)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=8, V=5)
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, np.zeros(8), p)
    assert out["loss"] == 0.0 and out["N"] == 0 and np.all(out["dlogits"] == 0.0)
    assert np.all(out["flags"] == 0)


def test_caller_denominator_and_grad_scale():
    rng = np.random.default_rng(70)
    z, ids, lp_old, lp_mu, adv = _tiny_batch(rng, T=20, V=6)
    base = decoupled_loss(z, ids, lp_old, lp_mu, adv, None, P)
    p2 = LossParams(0.5, 2.0, 0.2, 0.28, denom=80, grad_scale=3.0)
    out = decoupled_loss(z, ids, lp_old, lp_mu, adv, None, p2)
    assert abs(out["loss"] * 80 - base["loss"] * 20) < 1e-13
    np.testing.assert_allclose(out["dlogits"] * 80 / 3.0, base["dlogits"] * 20, atol=1e-15)


def test_proxy_ratio_closed_forms():
    """App. A: with the log-linear proxy r_d = r^(1-alpha) and r_s = r^alpha; with
    the arithmetic proxy r_d = alpha + (1 - alpha) r, where r = pi_theta / mu_old."""
    rng = np.random.default_rng(80)
    lmu = rng.normal(-4, 1, size=50)
    r = np.exp(rng.normal(0, 0.3, size=50))
    lth = lmu + np.log(r)
    for alpha in (0.25, 1 / 3, 0.5, 0.9):
        for kind in ("loglinear", "arithmetic"):
            lp = proxy_logprob(kind, alpha, lmu, lth)
            out = token_terms(lth, lp, lmu, np.ones(50), None, P)
            if kind == "loglinear":
                np.testing.assert_allclose(out["r_d"], r ** (1 - alpha), rtol=1e-12)
                np.testing.assert_allclose(out["r_s"], r ** alpha, rtol=1e-12)
            else:
                np.testing.assert_allclose(out["r_d"], alpha + (1 - alpha) * r, rtol=1e-12)
                np.testing.assert_allclose(out["r_s"], r / (alpha + (1 - alpha) * r), rtol=1e-12)
    # alpha = 0 gives pi_prox = pi_theta (r_s = 1); alpha = 1 gives mu_old (r_d = 1)
    for kind in ("loglinear", "arithmetic"):
        np.testing.assert_allclose(proxy_logprob(kind, 0.0, lmu, lth), lth, atol=1e-13)
        np.testing.assert_allclose(proxy_logprob(kind, 1.0, lmu, lth), lmu, atol=1e-13)


def test_thresholds_inclusive_at_the_exact_bound():
    """Eq. 4's M_[1/c,c] and Eq. 3's r_s <= 1 + eps (A >= 0) / r_s >= 1 - eps (A < 0)
    include the bound itself.  The bounds are chosen as exp(d) of the very
    log-ratio d the oracle will see, so the ratio equals the bound exactly."""
    lmu = np.array([-2.0, -2.0])
    d = np.array([0.125, -0.25])             # log r_d at the upper / lower band edge
    lold = lmu + d
    assert np.all(lold - lmu == d)
    p = LossParams(rd_lo=float(np.exp(d[1])), rd_hi=float(np.exp(d[0])), eps_low=0.2,
                   eps_high=0.28)
    out = token_terms(lold, lold, lmu, np.array([1.0, 1.0]), None, p)
    assert out["r_d"][0] == p.rd_hi and out["r_d"][1] == p.rd_lo
    assert np.all(out["in_band"])
    # clip bounds hit exactly: r_s = exp(ds) in [1, 2) so that 1 + (exp(ds) - 1) == exp(ds)
    ds, dl = 0.25, -0.125
    up = float(np.exp(ds))
    lo = float(np.exp(dl))
    lth = np.array([-3.0 + ds, -3.0 + dl])
    lold = np.array([-3.0, -3.0])
    assert np.all(lth - lold == np.array([ds, dl]))
    p = LossParams(rd_lo=0.5, rd_hi=2.0, eps_low=1.0 - lo, eps_high=up - 1.0)
    assert 1.0 + p.eps_high == up and 1.0 - p.eps_low == lo
    out = token_terms(lth, lold, lold, np.array([1.0, -1.0]), None, p)
    assert out["r_s"][0] == up and out["r_s"][1] == lo
    assert np.all(out["mis"]) and out["n_clipped"] == 0


def test_open_band_role_weights_by_the_total_ratio():
    # Table 5, "PPO-EWMA" row: r_2 * M(r_1) with no mask on r_2 (band [0, inf)).
    # With a clip interval too wide to bind, every token is active and its
    # weight is r_d * r_s = pi_theta / mu_old (the total ratio of Sec. 3.2), so
    # the token-mean loss is -sum(exp(log pi_theta - log mu) * A) / N, computed
    # here straight from the inputs.
    rng = np.random.default_rng(17)
    T = 64
    lt = rng.normal(-3.0, 1.0, T)
    lo = lt + rng.normal(0.0, 0.1, T)
    lm = lo + rng.normal(0.0, 1.5, T)       # r_d spread over two orders of magnitude
    A = rng.normal(0.0, 1.0, T)
    m = (rng.random(T) < 0.8).astype(np.uint8)
    p = LossParams(rd_lo=0.0, rd_hi=float("inf"), eps_low=1.0, eps_high=1e9, rd_weight=1)
    o = token_terms(lt, lo, lm, A, m, p)
    v = m.astype(bool)
    assert o["n_rd_out"] == 0 and o["n_active"] == o["n_valid"] == v.sum()
    expect = -math.fsum(np.exp(lt[v] - lm[v]) * A[v]) / v.sum()
    assert abs(o["loss"] - expect) <= 1e-12 * max(1.0, abs(expect))
    # without the r_d weight (rd_weight = 0) the same tokens weigh r_s alone
    o0 = token_terms(lt, lo, lm, A, m, LossParams(rd_lo=0.0, rd_hi=float("inf"), eps_low=1.0,
                                                  eps_high=1e9, rd_weight=0))
    expect0 = -math.fsum(np.exp(lt[v] - lo[v]) * A[v]) / v.sum()
    assert abs(o0["loss"] - expect0) <= 1e-12 * max(1.0, abs(expect0))


def test_threshold_distances_measure_to_the_deciding_edge():
    # The exemption from bit-exactness is decided by the distance, in log-ratio
    # space, to the threshold that decides the token: the clip edge of the
    # advantage's sign (log(1 + eps_high) for A >= 0, log(1 - eps_low) for A < 0)
    # and the nearer band edge.  Hand-built tokens at known distances.
    p = LossParams(0.5, 2.0, 0.2, 0.28)
    d = np.array([1e-7, -3e-7, 2e-3, -5e-4])
    edge_hi, edge_lo = np.log1p(0.28), np.log1p(-0.2)
    for A, edge in ((1.0, edge_hi), (0.0, edge_hi), (-1.0, edge_lo)):
        lt = edge + d                       # log pi_theta, with log pi_old = 0
        o = token_terms(lt, np.zeros(4), np.zeros(4), np.full(4, A), None, p)
        assert np.allclose(o["dist_rs"], np.abs(d), rtol=0, atol=1e-12), A
        assert np.allclose(o["dist_rd"], np.log(2.0), rtol=0, atol=1e-12)   # log r_d = 0
    for edge in (np.log(0.5), np.log(2.0)):
        lo_ = edge + d                      # log pi_old, with log mu_old = 0
        o = token_terms(lo_, lo_, np.zeros(4), np.ones(4), None, p)
        assert np.allclose(o["dist_rd"], np.abs(d), rtol=0, atol=1e-12), edge


def test_bad_ids_are_counted_among_unmasked_tokens_only():
    # Interface convention: a token whose id is outside [0, V) is dropped, and it
    # counts as a bad id only if the loss mask keeps it (a masked token carries
    # no evidence either way).
    z = np.zeros((4, 5))
    ids = np.array([1, 7, -1, 2])
    mask = np.array([1, 1, 0, 1], dtype=np.uint8)
    lt, _ = token_logprob(z, ids)
    o = token_terms(lt, lt, lt, np.ones(4), mask, LossParams(0.5, 2.0, 0.2, 0.28),
                    id_ok=(ids >= 0) & (ids < 5))
    assert o["bad_ids"] == 1 and o["n_valid"] == 2 and o["N"] == 2
