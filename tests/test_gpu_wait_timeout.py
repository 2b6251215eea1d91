"""Failure detection of the cluster kernels' bounded waits, without a GPU fault.

The TMA-pipelined K2 kernels wait on an mbarrier for each prefetched row
slice, with a wall-clock limit.  A test hook makes the producer skip one
row's copy (a flag that nothing sets): the consumers' wait must run out,
the call must still complete and report OCC_DATA_ERR_TIMEOUT in the stats,
and the context must stay usable (the next call, without the hook, is
correct).  Runs in a child process so the variant and hooks are its own.
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import os, sys, numpy as np, torch
sys.path.insert(0, {root!r}); sys.path.insert(0, {tests!r})
from oracle_runner import fp32, logprob_rows, loss_params, oracle_loss
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch
b = make_loss_batch("agentic_bf16_v151936", T=96, seed=3, device="cuda")
b.mask.fill_(1)
lo64, _ = logprob_rows(b.z_old, b.ids, np.arange(b.T))
lp_old = torch.from_numpy(fp32(lo64)).cuda()
os.environ["OCC_TEST_LOST_COPY_ROW"] = "5"
os.environ["OCC_TEST_WAIT_TIMEOUT_NS"] = "200000000"
out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                     **b.thresholds())
torch.cuda.synchronize()
st = occ.decode_loss_stats(out["stats"])
assert st.err & 2, st
del os.environ["OCC_TEST_LOST_COPY_ROW"], os.environ["OCC_TEST_WAIT_TIMEOUT_NS"]
out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                     **b.thresholds())
torch.cuda.synchronize()
st = occ.decode_loss_stats(out["stats"])
lt64, _ = logprob_rows(b.z_theta, b.ids, np.arange(b.T))
o = oracle_loss(b, lt64, fp32(lo64), loss_params(b))
assert st.err == 0 and abs(st.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
print("timeout ok")
"""


@pytest.mark.parametrize("variant", ["tma", "reg"])
def test_lost_copy_times_out_and_reports(variant):
    env = dict(os.environ, OCC_K2_VARIANT=variant)
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0 and "timeout ok" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
