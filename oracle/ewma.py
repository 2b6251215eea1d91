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
below tau.  App. D speaks of consecutive low-ratio streaks; the oracle counts
a streak and resets once it reaches ``min_streak`` (1 = reset on the first low
step, the Sec. 5.2 rule).  A step with no valid tokens carries no evidence:
the streak is left unchanged.
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
