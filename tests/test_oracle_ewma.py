"""Pins for the oracle's R10 (revised PPO-EWMA, Sec. 5.2, Eq. 5, App. B).

The App. B recursion is checked against the Eq. 5 closed form (a different
expression of the same average); the weights sum to one; the stationary
update is Table 1's plain EWMA; the center of mass and the W/(W+2) rule are
checked against numerically summed series; resets are exact.
"""

import math

import numpy as np
import pytest

from oracle import (EwmaState, beta_for_window, center_of_mass, ewma_closed_form,
                    ewma_coefficients, ewma_update)


@pytest.mark.parametrize("beta", [0.5, 0.75, 0.99])
def test_recursion_equals_closed_form(beta):
    rng = np.random.default_rng(1)
    thetas = [rng.normal(0, 0.02, size=64) for _ in range(10)]
    st = EwmaState()
    tp = np.zeros(64)
    for t, th in enumerate(thetas):
        tp, st, _ = ewma_update(tp, th, beta, st)
        np.testing.assert_allclose(tp, ewma_closed_form(thetas[:t + 1], beta), rtol=1e-13,
                                   atol=1e-16)
    assert abs(st.w - sum(beta ** k for k in range(10))) < 1e-12


def test_first_step_copies_and_weights_sum_to_one():
    a, b, reset, st = ewma_coefficients(EwmaState(), 0.9)
    assert (a, b, reset, st.w) == (0.0, 1.0, False, 1.0)
    st = EwmaState(w=3.7)
    for _ in range(20):
        a, b, _, st = ewma_coefficients(st, 0.8)
        assert abs(a + b - 1.0) < 1e-15


def test_constant_parameters_are_a_fixed_point():
    th = np.linspace(-1, 1, 33)
    st = EwmaState(w=5.0)
    tp = th.copy()
    for _ in range(5):
        tp, st, _ = ewma_update(tp, th, 0.93, st)
    np.testing.assert_allclose(tp, th, rtol=1e-15, atol=1e-16)


def test_stationary_limit_is_table1_plain_ewma():
    # Table 1: theta_prox,t = beta theta_prox,t-1 + (1 - beta) theta_t, which is
    # the recursion at its fixed point w = 1 / (1 - beta).
    beta = 0.99
    a, b, _, st = ewma_coefficients(EwmaState(w=1.0 / (1.0 - beta)), beta)
    assert abs(b - (1.0 - beta)) < 1e-15 and abs(a - beta) < 1e-15
    assert abs(st.w - 1.0 / (1.0 - beta)) < 1e-12


def test_center_of_mass_series_and_window_rule():
    for beta in (0.5, 0.75, 0.9, 0.99):
        k = np.arange(20000)
        w = beta ** k
        assert abs(math.fsum(k * w) / math.fsum(w) - center_of_mass(beta)) < 1e-9
    for W in (1, 2, 3, 6, 10):
        # the rule places the center of mass at the window midpoint W / 2
        assert abs(center_of_mass(beta_for_window(W)) - W / 2.0) < 1e-12
    assert beta_for_window(6) == 0.75


def test_reset_is_exact_and_counts():
    rng = np.random.default_rng(2)
    th = rng.normal(0, 0.02, size=100).astype(np.float32)
    tp = th + rng.normal(0, 1e-4, size=100).astype(np.float32)
    st = EwmaState(w=100.0, streak=0, n_resets=2)
    new, st2, (a, b, reset) = ewma_update(tp, th, 0.99, st, n_active=80, n_valid=100, tau=0.9)
    assert reset and np.array_equal(new, th.astype(np.float64))
    assert (st2.w, st2.streak, st2.n_resets) == (1.0, 0, 3)
    new, st3, (_, _, reset) = ewma_update(tp, th, 0.99, st, n_active=95, n_valid=100, tau=0.9)
    assert not reset and st3.streak == 0 and st3.n_resets == 2


def test_streak_rule():
    st = EwmaState(w=4.0)
    seq = [(50, 100), (99, 100), (50, 100), (50, 100), (10, 0), (50, 100)]
    resets = []
    for n_act, n_val in seq:
        _, _, reset, st = ewma_coefficients(st, 0.75, n_active=n_act, n_valid=n_val,
                                            tau=0.9, min_streak=2)
        resets.append((reset, st.streak))
    # low, high (streak cleared), low, low (second in a row: reset), no tokens
    # (no evidence, streak kept), low
    assert resets == [(False, 1), (False, 0), (False, 1), (True, 0), (False, 0), (False, 1)]
    _, _, reset, _ = ewma_coefficients(EwmaState(w=2.0), 0.75, force_reset=True)
    assert reset
    # Sec. 5.2 resets when rho < tau: rho exactly at tau does not count as low
    _, _, reset, st = ewma_coefficients(EwmaState(w=2.0), 0.75, n_active=9, n_valid=10, tau=0.9)
    assert 9 / 10 == 0.9 and not reset and st.streak == 0


# ---------------------------------------------------------------- bf16 buffers

def test_splitmix64_reference_outputs():
    # Reference outputs of SplitMix64 for seed 1234567, as printed by its public
    # reference implementation (Steele, Lea and Flood 2014; splitmix64.c).
    from oracle import splitmix64_at
    expect = [6457827717110365317, 3203168211198807973, 9817491932198370423,
              4593380528125082431, 16408922859458223821]
    assert [int(v) for v in splitmix64_at(1234567, np.arange(5))] == expect


def test_bf16_nearest_matches_torch_and_ties_to_even():
    torch = pytest.importorskip("torch")
    from oracle import round_bf16
    rng = np.random.default_rng(3)
    x = (rng.standard_normal(100000) * np.exp(rng.uniform(-20, 20, 100000))).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(round_bf16(x), ref)
    # exact midpoints: 1 + 2^-8 lies between 1 and 1 + 2^-7 -> even (1.0)
    mid = np.array([1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8], dtype=np.float32)
    out = round_bf16(mid)
    assert out[0] == 0x3F80 and out[1] == 0x3F82


def test_bf16_stochastic_rounding_is_unbiased_and_brackets():
    from oracle import bf16_bits_to_f32, round_bf16
    x = np.full(200000, 1.0 + 0.3 * 2.0 ** -7, dtype=np.float32)   # 30 % of a bf16 ulp above 1
    bits = round_bf16(x, seed=99, idx=np.arange(x.size, dtype=np.uint64))
    vals = bf16_bits_to_f32(bits)
    assert set(np.unique(vals).tolist()) == {1.0, 1.0 + 2.0 ** -7}
    frac = np.mean(vals > 1.0)
    assert abs(frac - 0.3) < 0.005                      # rounds up with the dropped fraction
    assert abs(vals.astype(np.float64).mean() - float(x[0])) < 2e-5
    neg = round_bf16(-x, seed=99, idx=np.arange(x.size, dtype=np.uint64))
    assert np.array_equal(neg, bits | 0x8000)          # magnitude rounding: sign symmetric


def test_bf16_step_tracks_float64_recursion():
    from oracle import bf16_bits_to_f32, ewma_update_bf16, round_bf16
    rng = np.random.default_rng(4)
    th = (rng.standard_normal(50000) * 0.02).astype(np.float32)
    tp = round_bf16((th + rng.standard_normal(50000) * 1e-3).astype(np.float32))
    exact = 0.25 * bf16_bits_to_f32(tp).astype(np.float64) + 0.75 * th
    out = bf16_bits_to_f32(ewma_update_bf16(tp, th, 0.75, copy=False)).astype(np.float64)
    ulp = np.abs(exact) * 2.0 ** -7
    assert np.all(np.abs(out - exact) <= 0.5 * ulp * (1 + 1e-3) + 1e-12)
    assert np.array_equal(ewma_update_bf16(tp, th, 1.0, copy=True), round_bf16(th))


def test_fma_f32_single_rounding():
    from fractions import Fraction
    from oracle.ewma import fma_f32
    rng = np.random.default_rng(5)
    a = rng.standard_normal(2000).astype(np.float32)
    b = (rng.standard_normal(2000) * 1e-3).astype(np.float32)
    c = rng.standard_normal(2000).astype(np.float32)
    # midpoint constructions: c + a*b lands exactly half a float32 ulp plus a tiny product
    c[:8] = np.float32(1.0)
    a[:8] = np.float32(2.0 ** -24)
    b[:8] = np.float32(1.0) + np.float32(2.0 ** -23) * np.arange(8, dtype=np.float32)
    # a*b = (1 + 2^-12)^2 = 1 + 2^-11 + 2^-24 is exactly a float32 midpoint, and a
    # tiny c (below float64 resolution at 1) makes the float64 sum land on it while
    # the exact value lies just above or below: only the sum's rounding error tells
    # which way to round (both signs, several scales)
    k = np.arange(8, 16)
    scale = np.float32(2.0) ** ((k % 4) - 2).astype(np.float32)
    a[8:16] = (np.float32(1.0) + np.float32(2.0 ** -12)) * scale
    b[8:16] = np.float32(1.0) + np.float32(2.0 ** -12)
    c[8:16] = np.where(k % 2 == 0, 1.0, -1.0).astype(np.float32) * np.float32(2.0 ** -60) * scale
    got = fma_f32(a, b, c)
    for i in range(2000):
        exact = Fraction(float(a[i])) * Fraction(float(b[i])) + Fraction(float(c[i]))
        lo = np.float32(float(exact))
        # correctly rounded float32 of the exact value: compare against both neighbours
        cands = [lo, np.nextafter(lo, np.float32(np.inf)), np.nextafter(lo, np.float32(-np.inf))]
        best = min(cands, key=lambda x: (abs(Fraction(float(x)) - exact),
                                        int(np.float32(x).view(np.uint32)) & 1))
        assert got[i] == best, i


def test_bf16_rounding_keeps_infinities_and_nans():
    # inf stays inf and NaN stays NaN (sign kept) under both roundings, whatever
    # the payload: adding the rounding increment to a NaN whose mantissa bits are
    # all set would carry into the sign bit and give a zero.  Finite values at the
    # top of the range round to the largest bf16 or to inf as float32 -> bf16
    # rounding to nearest does (torch's conversion).
    torch = pytest.importorskip("torch")
    from oracle import round_bf16
    bits = np.array([0x7F800000, 0xFF800000, 0x7FC00000, 0x7FFFFFFF, 0xFFFFFFFF, 0x7F800001,
                     0xFFC00001], dtype=np.uint32)
    x = bits.view(np.float32)
    for seed in (0, 1, 77, 2 ** 40 + 3):
        out = round_bf16(x, seed, np.arange(x.size, dtype=np.uint64))
        exp_all_ones = (out & 0x7F80) == 0x7F80
        assert np.all(exp_all_ones), (seed, [hex(v) for v in out])
        assert np.all((out & 0x8000) == ((bits >> 16) & 0x8000)), seed      # sign kept
        assert np.all(((out & 0x7F) != 0) == np.isnan(x)), seed              # NaN iff NaN
    big = np.array([3.3895e38, 3.39e38, 3.4e38, -3.4e38], dtype=np.float32)
    want = torch.from_numpy(big).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(round_bf16(big, 0), want)
