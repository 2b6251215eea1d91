"""Float64 oracle of the revised PPO-EWMA proximal parameters (rule R10).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Sec. 5.2, Eq. 5: theta_prox^(t) = sum_k beta^(t-k) theta^(k) / sum_k beta^(t-k),
and pi_prox replaces the missing pi_old in both r_s and r_d.
App. B gives the same quantity as a recursion on a cumulative weight:
    w^(t) = 1 + beta w^(t-1),
    theta_prox^(t) = theta^(t) / w^(t) + beta (w^(t-1) / w^(t)) theta_prox^(t-1),
with w^(-1) = 0 for an empty history.  In the stationary limit w -> 1/(1-beta)
and the update is the plain EWMA of Table 1 (b = 1 - beta).
Sec. 5.2 also sets beta ~ W/(W+2) for a staleness window W (center of mass of
the history, App. B) and resets theta_prox <- theta^(t) when the Train-Infer
Mask value rho_t (fraction of tokens active after masking and clipping) drops
below tau.  App. E speaks of consecutive low-ratio streaks; the oracle counts
a streak and resets once it reaches ``min_streak`` (1 = reset on the first low
step, the Sec. 5.2 rule).  A step with no valid tokens carries no evidence:
the streak is left unchanged.

A bf16 proximal buffer (the footprint of the paper's host-side copy, Table 3a)
is modelled in the kernel's precision, see ``ewma_update_bf16``.
"""

from dataclasses import dataclass, replace

import numpy as np


@dataclass
class EwmaState:
    """w = w^(t-1) (0 for an empty history); streak = consecutive low-rho steps."""
    w: float = 0.0
    streak: int = 0
    n_resets: int = 0


def ewma_coefficients(state, beta, n_active=None, n_valid=None, tau=0.9, min_streak=1,
                      force_reset=False):
    """One step of the App. B recursion plus the Sec. 5.2 auto-reset rule.

    Returns (a, b, reset, new_state) such that the new proximal parameters are
    a * theta_prox + b * theta (a = beta w^(t-1)/w^(t), b = 1/w^(t)), or exactly
    theta when ``reset`` is True.
    """
    streak = state.streak
    if n_valid is not None and n_valid > 0:
        rho = n_active / n_valid
        streak = streak + 1 if rho < tau else 0
    reset = bool(force_reset) or (n_valid is not None and n_valid > 0 and streak >= min_streak)
    if reset:
        return 0.0, 1.0, True, EwmaState(w=1.0, streak=0, n_resets=state.n_resets + 1)
    w_prev = float(state.w)
    w = 1.0 + beta * w_prev
    a = beta * w_prev / w
    b = 1.0 / w
    return a, b, False, replace(state, w=w, streak=streak)


def ewma_update(theta_prox, theta, beta, state, **reset_args):
    """theta_prox^(t) from theta_prox^(t-1) and theta^(t) (App. B; reset of Sec. 5.2).

    Returns (new_theta_prox float64 array, new_state, (a, b, reset)).
    """
    a, b, reset, st = ewma_coefficients(state, beta, **reset_args)
    tp = np.asarray(theta_prox, dtype=np.float64)
    th = np.asarray(theta, dtype=np.float64)
    new = th.copy() if reset else a * tp + b * th
    return new, st, (a, b, reset)


def ewma_closed_form(thetas, beta):
    """Eq. 5: normalised exponentially weighted average of theta^(0..t)."""
    t = len(thetas) - 1
    num = sum(beta ** (t - k) * np.asarray(th, dtype=np.float64) for k, th in enumerate(thetas))
    den = sum(beta ** (t - k) for k in range(t + 1))
    return num / den


def beta_for_window(W):
    """Sec. 5.2 / App. B: beta ~ W/(W+2) puts the history's center of mass at W/2."""
    return W / (W + 2.0)


def center_of_mass(beta):
    """App. B: stationary center of mass of the EWMA history, beta / (1 - beta)."""
    return beta / (1.0 - beta)


# --------------------------------------------------------------- bf16 buffers
#
# For a bf16 proximal buffer the stored value is a quantised code, so the
# oracle takes the rounding decision in the kernel's precision: the update is
# formed in float32 (one rounding of theta - theta_prox, one fused
# multiply-add), then rounded to bf16 by definition: nearest with ties to even,
# or stochastically with the bits of a SplitMix64 counter stream.

_GAMMA = np.uint64(0x9E3779B97F4A7C15)


def splitmix64_at(seed, i):
    """The i-th output (i >= 0) of SplitMix64 started at `seed` (Steele, Lea and
    Flood, 2014): state_i = seed + (i + 1) gamma, output = mix(state_i)."""
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (np.asarray(i, dtype=np.uint64) + np.uint64(1)) * _GAMMA
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        return z ^ (z >> np.uint64(31))


def bf16_bits_to_f32(bits):
    return (np.asarray(bits, dtype=np.uint32) << np.uint32(16)).view(np.float32)


def sr_bits(seed, idx):
    """16 random bits for parameter idx: lane (idx mod 4) of the (idx // 4)-th
    SplitMix64 output, lane 0 being the least significant 16 bits."""
    idx = np.asarray(idx, dtype=np.uint64)
    out = splitmix64_at(seed, idx >> np.uint64(2))
    return (out >> (np.uint64(16) * (idx & np.uint64(3)))) & np.uint64(0xFFFF)


def round_bf16(x32, seed=0, idx=None):
    """float32 -> bf16 bits.  seed == 0: nearest, ties to even.  Otherwise add 16
    random bits (``sr_bits``) below the bf16 unit in the last place and
    truncate (stochastic rounding of the magnitude).  Infinities are exact; a
    NaN rounds to a quiet NaN of the same sign (0x7FC0 with the sign bit), as
    rounding must keep a NaN a NaN whatever bits its payload holds."""
    u = np.asarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    special = (u & np.uint64(0x7F800000)) == np.uint64(0x7F800000)
    nan = special & ((u & np.uint64(0x007FFFFF)) != np.uint64(0))
    if seed == 0:
        lsb = (u >> np.uint64(16)) & np.uint64(1)
        r = np.uint64(0x7FFF) + lsb
    else:
        r = sr_bits(seed, idx)
    out = ((u + r) >> np.uint64(16)) & np.uint64(0xFFFF)
    trunc = (u >> np.uint64(16)) & np.uint64(0xFFFF)          # exact for the infinities
    quiet = ((u >> np.uint64(16)) & np.uint64(0x8000)) | np.uint64(0x7FC0)
    return np.where(nan, quiet, np.where(special, trunc, out)).astype(np.uint16)


def fma_f32(a, b, c):
    """float32 fused multiply-add a * b + c, rounded once to nearest-even.

    The product of two float32 values is exact in float64; the float64 sum is
    exact up to its TwoSum error e.  Rounding s = fl64(p + c) to float32 is
    then correct except when s falls exactly on a float32 midpoint, where the
    sign of e decides the side."""
    # (for an infinite or NaN operand the TwoSum terms are NaN, the midpoint test
    # is false and r is the float32 of s: inf or NaN, as a fused multiply-add gives)
    with np.errstate(invalid="ignore"):
        p = np.asarray(a, np.float64) * np.asarray(b, np.float64)
        c = np.asarray(c, np.float64)
        s = p + c
        bp = s - p
        e = (p - (s - bp)) + (c - bp)              # TwoSum: p + c = s + e exactly
        r = s.astype(np.float32)
        d = s - r.astype(np.float64)               # exact
        half = np.spacing(np.abs(r)).astype(np.float64) / 2
        fix = (np.abs(d) == half) & (d * e > 0)    # past the midpoint: round away from r
        r = np.where(fix, np.nextafter(r, np.where(d > 0, np.float32(np.inf), np.float32(-np.inf))),
                     r)
    return r.astype(np.float32)


def ewma_update_bf16(tp_bits, theta32, b, copy, seed=0, idx0=0):
    """One App. B step on a bf16 buffer in the kernel's precision:
    v = fma(b, theta - tp, tp) in float32 (or theta itself on a reset / first
    step), rounded to bf16."""
    tp = bf16_bits_to_f32(tp_bits)
    th = np.asarray(theta32, dtype=np.float32)
    with np.errstate(invalid="ignore"):            # signalling-NaN parameters stay NaN
        v = th if copy else fma_f32(np.float32(b), (th - tp).astype(np.float32), tp)
    idx = np.arange(idx0, idx0 + tp.size, dtype=np.uint64)
    return round_bf16(v, seed, idx)
