"""Float64 oracle of the interpolation proxies for a missing pi_old (rule R12).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Table 1 lists proxy references built per token from the rollout policy
mu_old and the current policy pi_theta, with behaviour-policy weight alpha;
App. A analyses them (Proposition 1):
    log-linear:  log pi_prox = alpha log mu_old + (1 - alpha) log pi_theta
    arithmetic:  pi_prox = alpha mu_old + (1 - alpha) pi_theta   ("linear_prox")
The proxy then stands in for pi_old in r_d = pi_prox / mu_old and
r_s = pi_theta / pi_prox.  It is a constant of the objective (its gradient is
not taken), so R8 is unchanged.
"""

import numpy as np

KINDS = ("loglinear", "arithmetic")


def proxy_logprob(kind, alpha, logp_mu, logp_theta):
    """log pi_prox(y_t) per token (Table 1, App. A)."""
    lm = np.asarray(logp_mu, dtype=np.float64)
    lt = np.asarray(logp_theta, dtype=np.float64)
    if kind == "loglinear":
        return alpha * lm + (1.0 - alpha) * lt
    if kind == "arithmetic":
        return np.log(alpha * np.exp(lm) + (1.0 - alpha) * np.exp(lt))
    raise ValueError(kind)
