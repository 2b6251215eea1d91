"""Failure detection of the ring kernel's bounded waits, without a GPU fault.

The persistent TMA-ring fused kernel (option fused_variant = 1) waits on
mbarriers for every copy it issues, each wait limited in wall-clock time.  A
test control makes its producer take a ring slot for one copy of one row
without issuing the copy (nothing will ever complete that phase): the
consumers' wait must run out, every other wait must give up on the CTA's
abort flag, the producer must drain the copies it did issue, and the call
must report OCC_DATA_ERR_TIMEOUT in the stats.  The context must stay usable:
the next call, without the control, matches the oracle.
"""

import numpy as np
import pytest
import torch

from oracle_runner import logprob_rows, loss_params, oracle_loss
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu


def test_lost_copy_times_out_and_reports():
    b = make_loss_batch("agentic_bf16_v151936", T=96, seed=3, device="cuda")
    b.mask.fill_(1)
    args = (b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask)
    with occ.options(fused_variant=1, test_lost_copy_row=5, test_wait_ns=200_000_000):
        out = occ.occ_decoupled_loss_fused(*args, **b.thresholds())
        assert occ.occ_last_kernel() == "k2_fused_ring"
        torch.cuda.synchronize()
    st = occ.decode_loss_stats(out["stats"])
    assert st.err & occ.DATA_ERR_TIMEOUT, st
    with occ.options(fused_variant=1):
        out = occ.occ_decoupled_loss_fused(*args, **b.thresholds())
        torch.cuda.synchronize()
    st = occ.decode_loss_stats(out["stats"])
    rows = np.arange(b.T)
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, _ = logprob_rows(b.z_theta, b.ids, rows)
    o = oracle_loss(b, lt64, lo64, loss_params(b))
    assert st.err == 0 and st.n_valid == o["n_valid"]
    assert abs(st.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
