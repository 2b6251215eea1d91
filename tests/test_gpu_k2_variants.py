"""The alternative K2 kernels (selected with OCC_K2_VARIANT) against the oracle.

The default K2 kernel is the two-pass L2 kernel; the cluster kernels
("tma": persistent cp.async.bulk pipeline with the row slice in shared memory,
"reg": register-resident terms) and the 1024-thread L2 kernel are kept as
tuning alternatives.  The variant is read once per process, so each runs in a
child process on a few workloads, comparing with the oracle.
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys, numpy as np, torch
sys.path.insert(0, {root!r}); sys.path.insert(0, {tests!r})
from oracle_runner import fp32, logprob_rows, loss_params, oracle_loss, dlogits_rows
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch
for name, T, f32 in (("agentic_bf16_v151936", 200, False), ("grpo_bf16_v32000", 300, True),
                     ("tiny_f32_v4096", 256, False)):
    b = make_loss_batch(name, T=T, seed=7, device="cuda")
    rows = np.arange(b.T)
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    o = oracle_loss(b, lt64, fp32(lo64), loss_params(b))
    out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, torch.from_numpy(fp32(lo64)).cuda(),
                                         b.logp_mu, b.adv, b.mask, dlogits_f32=f32, **b.thresholds())
    torch.cuda.synchronize()
    s = occ.decode_loss_stats(out["stats"])
    fl = out["flags"].cpu().numpy()
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    assert not ((fl != o["flags"]) & ~near).any(), name
    assert abs(s.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12, name
    v = o["valid"]
    assert np.abs(out["logp"].cpu().numpy()[v] - lt64[v]).max() <= 1e-5, name
    pick = np.unique(np.concatenate([np.nonzero(o["g"])[0][:12], [0, b.T - 1]]))
    ref = dlogits_rows(b, pick, lse[pick], o["g"][pick])
    got = out["dlogits"][torch.as_tensor(pick, device="cuda")].float().cpu().numpy()
    g = np.abs(o["g"][pick])[:, None]
    rel = 2e-6 if (f32 or b.z_theta.dtype == torch.float32) else 2.0 ** -8
    assert np.all(np.abs(got - ref) <= rel * np.abs(ref) + 4e-6 * g + 1e-30), name
print("variant ok")
"""


@pytest.mark.parametrize("variant", ["tma", "reg", "l2_1024"])
def test_k2_variant_against_oracle(variant):
    env = dict(os.environ, OCC_K2_VARIANT=variant)
    code = CHILD.format(root=ROOT, tests=os.path.join(ROOT, "tests"))
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and "variant ok" in r.stdout, r.stdout[-2000:] + r.stderr[-4000:]
