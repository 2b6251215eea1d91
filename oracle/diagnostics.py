"""Float64 oracle of per-token diagnostics of the proximal reference (rule R11).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Sec. 5.2, Sec. 6.5 and App. E describe the failure mode the revised PPO-EWMA guards
against: the reference policy drifts away from the policies that generated
recent rollouts (reference-policy lag), which shows up as a collapsing
Train-Infer Mask.  Two per-token quantities measure that lag directly from
the same logits rows the loss reads:
    H(pi_theta)            = - sum_v p_v log p_v,            p = softmax(z)
    KL(pi_old || pi_theta) =   sum_v q_v (log q_v - log p_v), q = softmax(z_old)
Both are the textbook definitions, written out here row by row.
"""

import numpy as np


def _log_softmax(z):
    z = np.asarray(z, dtype=np.float64)
    M = z.max(axis=1, keepdims=True)
    return z - (M + np.log(np.exp(z - M).sum(axis=1, keepdims=True)))


def token_entropy(z):
    """H(softmax(z[t])) for each row t."""
    lp = _log_softmax(z)
    return -(np.exp(lp) * lp).sum(axis=1)


def token_kl(z_old, z):
    """KL(softmax(z_old[t]) || softmax(z[t])) for each row t."""
    lq = _log_softmax(z_old)
    lp = _log_softmax(z)
    return (np.exp(lq) * (lq - lp)).sum(axis=1)
