"""Float64 CPU oracle for the decoupled off-policy correction path.

TEST INFRASTRUCTURE ONLY.  This package is the slow, plain reference that the
CUDA library is checked against.  Only the test suite, the smoke check in
``__graft_entry__`` and the ``cpu_baseline`` / ``--impl reference`` legs of
``bench.py`` may import it.  The product path (the C-ABI library and its Python
binding) never imports, calls or links anything here, and nothing here imports
the product package: the two share no code.  Inputs reach both sides from the
seeded generators in ``paper_2605_12070_gb300.workloads``, which hold none of
the method's arithmetic.

Every function follows a passage of the paper ("Missing Old Logits in
Asynchronous Agentic RL", arXiv 2605.12070) and cites it by section, equation or
table.  Arithmetic is numpy float64 on the exact (upcast) values of the inputs
the GPU sees.  Rows are processed in caller-chosen chunks; ``oracle.rows`` holds
the chunk/thread driver used for large inputs.

Modules
-------
loss   -- R1..R9: logsumexp/log-prob (Eq. 1 factors), the r_d band mask (Eq. 4),
          the sign-dependent PPO clip (Eqs. 2-3), token-mean loss, gradient.
ewma   -- R10: the revised PPO-EWMA proximal parameters (Eq. 5, App. B),
          the staleness-aware decay rule and the auto-reset rule (Sec. 5.2).
proxies -- R12: the log-linear and arithmetic interpolation proxies of
          Table 1 / App. A that stand in for a missing pi_old.
diagnostics -- R11: per-token entropy of pi_theta and KL(pi_old || pi_theta),
          the reference-lag diagnostics (Sec. 5.2, App. E).
rows   -- chunking / threading driver (no arithmetic of the method).

Pins: every function here is pinned by ``tests/test_oracle_*.py`` against
closed forms, invariants, brute force on tiny inputs, finite differences, and
the values printed in Table 4 (``tests/golden/``).  No function is unpinned.
"""

from .loss import LossParams, token_logprob, token_terms, decoupled_loss, softmax_grad_rows, \
    FLAG_IN_BAND, \
    FLAG_CLIPPED, FLAG_ACTIVE, FLAG_VALID  # noqa: F401
from .diagnostics import token_entropy, token_kl  # noqa: F401
from .proxies import proxy_logprob  # noqa: F401
from .ewma import EwmaState, ewma_coefficients, ewma_update, ewma_closed_form, \
    beta_for_window, center_of_mass, splitmix64_at, round_bf16, bf16_bits_to_f32, \
    ewma_update_bf16  # noqa: F401
