"""Float64 oracle of the decoupled correction loss (rules R1..R9).

TEST INFRASTRUCTURE ONLY (see the package docstring): the product path never
imports this module.

Notation follows the paper: mu_old is the inference-side rollout policy,
pi_old the training-side policy at the rollout version (or its stand-in
pi_prox / pi_async, Table 1), pi_theta the current policy, A_t the advantage.

R1  lse[t] = M + log sum_v exp(z[t,v] - M), M = max_v z[t,v];
    log pi(y_t) = z[t, y_t] - lse[t]                     (Eq. 1 factors)
R2  r_d = pi_old / mu_old; in band iff lo <= r_d <= hi   (Eq. 4, M_[1/c,c] is
    inclusive on both sides; Sec. 3.2)
R3  r_s = pi_theta / pi_old                              (Sec. 3.2, Eq. 1)
R4  MIS_ppo = 1{A>=0} 1{r_s <= 1+eps_high} + 1{A<0} 1{r_s >= 1-eps_low}
                                                         (Eq. 3; asymmetric
    thresholds as in App. A, "Numerical effective thresholds")
R5  w_d = r_d (Table 5 role "PPO-EWMA & train_infer": M(r2) r2 M(r1)) or
    w_d = 1   (Table 5 role "decoupled PPO & train_infer": M(r2) M(r1));
    r_d does not depend on theta, so w_d is a constant in the gradient.
R6  s_t = min(r_s A, clip(r_s, 1-eps_low, 1+eps_high) A);
    loss_t = - m_t M_d w_d s_t                           (Eq. 2 with the Eq. 4 mask)
R7  N = sum_t m_t; L = sum_t loss_t / N; N = 0 gives L = 0 (token mean)
R8  g_t = - grad_scale m_t M_d MIS_ppo w_d r_s A_t / N;
    dL/dz[t,v] = g_t (1[v = y_t] - softmax(z_theta[t])_v)
                                                         (the MIS gradient form
    stated after Eq. 2: MIS * r * A * grad log pi, with r = r_d r_s)
R9  n_valid = sum m; n_rd_out = sum m (1-M_d); n_clipped = sum m (1-MIS_ppo);
    n_active = sum m M_d MIS_ppo; the Train-Infer Mask value of Sec. 5.2 is
    rho = n_active / n_valid.

Token validity: m_t = loss_mask[t] != 0 and 0 <= y_t < V.  A token whose id is
out of range is dropped (treated as m_t = 0) and reported through ``bad_ids``;
this is an interface convention, not part of the paper.
"""

from dataclasses import dataclass

import numpy as np

FLAG_IN_BAND = 1   # r_d inside [lo, hi]
FLAG_CLIPPED = 2   # PPO clip active (not MIS_ppo)
FLAG_ACTIVE = 4    # m * M_d * MIS_ppo
FLAG_VALID = 8     # m (mask set and id in range)


@dataclass
class LossParams:
    """Thresholds and options of the decoupled loss.

    rd_lo, rd_hi   inclusive band on r_d (Eq. 4 uses [1/c, c]).
    eps_low/high   clip interval [1 - eps_low, 1 + eps_high] on r_s (Eq. 3, App. A).
    rd_weight      1: w_d = r_d (Table 5, PPO-EWMA & train_infer); 0: w_d = 1.
    grad_scale     upstream d(objective)/d(loss), multiplies the gradient only.
    denom          > 0: token-mean denominator given by the caller; else N = sum m.
    """
    rd_lo: float
    rd_hi: float
    eps_low: float
    eps_high: float
    rd_weight: int = 1
    grad_scale: float = 1.0
    denom: int = 0


def token_logprob(z, ids):
    """R1: per-row logsumexp and the log-probability of the sampled token.

    z   : (T, V) array, upcast exactly to float64.
    ids : (T,) integer token ids y_t.
    Returns (logp, lse), both float64 (T,).  logp is NaN where the id is
    outside [0, V).  (Eq. 1: each ratio is a quotient of such token
    probabilities.)
    """
    z = np.asarray(z, dtype=np.float64)
    ids = np.asarray(ids).astype(np.int64)
    T, V = z.shape
    if T == 0:
        return np.zeros(0), np.zeros(0)
    M = z.max(axis=1)
    lse = M + np.log(np.exp(z - M[:, None]).sum(axis=1))
    ok = (ids >= 0) & (ids < V)
    logp = np.full(T, np.nan)
    rows = np.nonzero(ok)[0]
    logp[rows] = z[rows, ids[rows]] - lse[rows]
    return logp, lse


def token_terms(logp_theta, logp_old, logp_mu, adv, mask, params, id_ok=None, N=None):
    """R2..R9 on per-token log-probabilities.

    logp_theta : log pi_theta(y_t)   (R1 on the current logits)
    logp_old   : log pi_old(y_t)     (or of pi_prox / pi_async, Table 1)
    logp_mu    : log mu_old(y_t)     (inference-side, an input)
    adv        : A_t
    mask       : loss mask m_t (None = all ones)
    id_ok      : per-token id validity (None = all valid)
    N          : token-mean denominator override (used when the caller splits
                 rows into chunks; default per R7 / params.denom)

    Returns a dict with per-token arrays (log_rd, log_rs, r_d, r_s, in_band,
    mis, valid, loss_t, g, flags, dist_rd, dist_rs) and scalars (N, loss_sum,
    loss, n_valid, n_rd_out, n_clipped, n_active, bad_ids).
    dist_rd / dist_rs are the distances |log r - log bound| to the nearest
    threshold that decides the token, in log-ratio space.
    """
    p = params
    lt = np.asarray(logp_theta, dtype=np.float64)
    lo_ = np.asarray(logp_old, dtype=np.float64)
    lm = np.asarray(logp_mu, dtype=np.float64)
    A = np.asarray(adv, dtype=np.float64)
    T = lt.shape[0]
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    ok = np.ones(T, dtype=bool) if id_ok is None else np.asarray(id_ok, dtype=bool)
    valid = m & ok
    bad_ids = int(np.sum(m & ~ok))

    # R2: discrepancy ratio and its inclusive band (ratio space, float64).
    log_rd = lo_ - lm
    r_d = np.exp(log_rd)
    in_band = (p.rd_lo <= r_d) & (r_d <= p.rd_hi)

    # R3: staleness ratio (set to 1 on dropped tokens, whose terms are unused).
    log_rs = np.where(valid, lt - lo_, 0.0)
    r_s = np.exp(log_rs)

    # R4: sign-dependent PPO active mask; A = 0 takes the A >= 0 branch.
    mis = np.where(A >= 0, r_s <= 1.0 + p.eps_high, r_s >= 1.0 - p.eps_low)

    # R5: role of r_d in the weight.
    w_d = r_d if p.rd_weight else np.ones(T)

    # R6: clipped surrogate and per-token loss.
    s = np.minimum(r_s * A, np.clip(r_s, 1.0 - p.eps_low, 1.0 + p.eps_high) * A)
    keep = valid & in_band
    loss_t = np.where(keep, -w_d * s, 0.0)

    # R7: token-mean denominator.
    if N is None:
        N = int(p.denom) if p.denom > 0 else int(np.sum(valid))
    loss_sum = float(np.sum(loss_t))
    loss = loss_sum / N if N > 0 else 0.0

    # R8 (scalar part): per-token gradient coefficient g_t.
    active = keep & mis
    if N > 0:
        g = np.where(active, -p.grad_scale * w_d * r_s * A / N, 0.0)
    else:
        g = np.zeros(T)

    # R9: counters and flags.
    flags = (in_band * FLAG_IN_BAND + (~mis) * FLAG_CLIPPED
             + active * FLAG_ACTIVE + FLAG_VALID).astype(np.uint8)
    flags = np.where(valid, flags, 0).astype(np.uint8)

    # distance (in log space) to the nearer band edge; an open edge (rd_lo = 0 or
    # rd_hi = inf: Table 5's unmasked r_2 roles) is infinitely far
    log_lo = np.log(p.rd_lo) if p.rd_lo > 0 else -np.inf
    log_hi = np.log(p.rd_hi) if np.isfinite(p.rd_hi) else np.inf
    dist_rd = np.minimum(np.abs(log_rd - log_lo), np.abs(log_rd - log_hi))
    log_clip_lo = np.log1p(-p.eps_low) if p.eps_low < 1.0 else -np.inf  # eps_low = 1: no lower edge
    dist_rs = np.where(A >= 0, np.abs(log_rs - np.log1p(p.eps_high)), np.abs(log_rs - log_clip_lo))
    return dict(
        log_rd=log_rd, log_rs=log_rs, r_d=r_d, r_s=r_s, in_band=in_band, mis=mis,
        valid=valid, loss_t=loss_t, g=g, flags=flags, dist_rd=dist_rd, dist_rs=dist_rs,
        N=N, loss_sum=loss_sum, loss=loss,
        n_valid=int(np.sum(valid)), n_rd_out=int(np.sum(valid & ~in_band)),
        n_clipped=int(np.sum(valid & ~mis)), n_active=int(np.sum(active)),
        bad_ids=bad_ids,
    )


def softmax_grad_rows(z, ids, lse, g):
    """R8 (vocabulary part): dL/dz[t,v] = g_t (1[v = y_t] - exp(z[t,v] - lse[t])).

    Rows with g_t = 0 (masked, out of band, clipped, A = 0 or invalid id) are
    exactly zero.
    """
    z = np.asarray(z, dtype=np.float64)
    T, V = z.shape
    g = np.asarray(g, dtype=np.float64)
    ids = np.asarray(ids).astype(np.int64)
    out = np.zeros((T, V))
    rows = np.nonzero(g != 0.0)[0]
    if rows.size:
        out[rows] = -g[rows, None] * np.exp(z[rows] - np.asarray(lse)[rows, None])
        out[rows, ids[rows]] += g[rows]
    return out


def decoupled_loss(z_theta, ids, logp_old, logp_mu, adv, mask, params, want_dlogits=True):
    """R1..R9 end to end on one batch held in memory.

    Returns the ``token_terms`` dict plus 'logp' (log pi_theta(y_t)), 'lse',
    and 'dlogits' (float64 (T, V)) when requested.
    """
    z = np.asarray(z_theta, dtype=np.float64)
    T, V = z.shape
    ids = np.asarray(ids).astype(np.int64)
    logp, lse = token_logprob(z, ids)
    id_ok = (ids >= 0) & (ids < V)
    out = token_terms(logp, logp_old, logp_mu, adv, mask, params, id_ok=id_ok)
    out["logp"] = logp
    out["lse"] = lse
    if want_dlogits:
        out["dlogits"] = softmax_grad_rows(z, np.where(id_ok, ids, 0), lse, out["g"])
    return out
