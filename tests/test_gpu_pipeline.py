"""HostFedStep: steps fed from pinned host memory, copies overlapping kernels.

Each step gets DIFFERENT inputs (a new batch of logits and token arrays, new
actor parameters), so a copy that overwrote a device buffer before the
previous step's kernels had read it would change that step's results.  The
pipelined steps must reproduce, bit for bit, the same steps run one after the
other from device-resident inputs (the kernels are deterministic).
"""

import pytest
import torch

from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.pipeline import HostFedStep
from paper_2605_12070_gb300.workloads import make_ewma_buffers, make_loss_batch

pytestmark = pytest.mark.gpu

STEPS = 3
N_PARAMS = 3_000_017


def _batches():
    bs = [make_loss_batch("agentic_bf16_v151936", T=384, seed=40 + k, device="cuda")
          for k in range(STEPS)]
    thetas = [make_ewma_buffers(N_PARAMS, seed=40 + k, device="cuda")[0] for k in range(STEPS)]
    return bs, thetas


def _loss_inputs(b):
    return [b.z_old, b.z_theta, b.ids, b.logp_mu, b.adv, b.mask]


@pytest.mark.parametrize("host_alloc", ["occ_host_alloc", "torch_pinned"])
def test_pipelined_steps_match_serial_steps(host_alloc):
    bs, thetas = _batches()
    b0 = bs[0]
    T, V = b0.T, b0.V
    thr = b0.thresholds()
    theta_prox0 = make_ewma_buffers(N_PARAMS, seed=99, device="cuda")[1]

    def outputs():
        return {"dl": torch.empty((T, V), dtype=torch.bfloat16, device="cuda"),
                "stats": occ.new_loss_stats("cuda"), "ws": occ.new_workspace(T, V, "cuda"),
                "tp": theta_prox0.clone(), "st": occ.new_ewma_state("cuda", w0=3.0)}

    def make_fns(inputs, theta, o):
        def loss():
            z_old, z_theta, ids, logp_mu, adv, mask = inputs
            occ.occ_decoupled_loss_fused(z_theta, z_old, ids, logp_mu, adv, mask, **thr,
                                         dlogits=o["dl"], stats=o["stats"], workspace=o["ws"])

        def ewma():
            occ.occ_ewma_update(o["tp"], theta, 0.9, o["st"], stats=o["stats"], tau=0.5)
        return loss, ewma

    # serial reference: device-resident inputs, one step after the other
    ref = outputs()
    ref_stats, ref_dl = [], []
    for k in range(STEPS):
        loss, ewma = make_fns(_loss_inputs(bs[k]), thetas[k], ref)
        loss()
        ewma()
        ref_stats.append(ref["stats"].clone())
        ref_dl.append(ref["dl"].clone())
    torch.cuda.synchronize()

    # pipelined: one set of device buffers, host inputs copied in every step
    def host_copy(t):
        if host_alloc == "occ_host_alloc":
            h = occ.occ_host_alloc(tuple(t.shape), t.dtype)
        else:
            h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h

    host_inputs = [[host_copy(t) for t in _loss_inputs(b)] for b in bs]
    host_thetas = [host_copy(t) for t in thetas]
    dev_inputs = [torch.empty_like(t) for t in _loss_inputs(b0)]
    dev_theta = torch.empty_like(thetas[0])
    out = outputs()
    kept_stats = [torch.empty_like(out["stats"]) for _ in range(STEPS)]
    kept_dl = [torch.empty_like(out["dl"]) for _ in range(STEPS)]
    k_done = [0]

    def keep():
        k = k_done[0]
        kept_stats[k].copy_(out["stats"], non_blocking=True)
        kept_dl[k].copy_(out["dl"], non_blocking=True)
        k_done[0] += 1

    loss, ewma = make_fns(dev_inputs, dev_theta, out)
    pipe = HostFedStep(dev_inputs, dev_theta, loss, ewma, after_step=keep)
    for k in range(STEPS):
        pipe.step(host_inputs[k], host_thetas[k])
    torch.cuda.synchronize()

    for k in range(STEPS):
        assert torch.equal(kept_stats[k], ref_stats[k]), k
        assert torch.equal(kept_dl[k], ref_dl[k]), k
    assert torch.equal(out["tp"], ref["tp"])
    assert torch.equal(out["st"], ref["st"])


def test_rejects_pageable_or_mismatched_host_inputs():
    b = make_loss_batch("agentic_bf16_v151936", T=64, seed=1, device="cuda")
    theta = torch.zeros(16, device="cuda")
    pipe = HostFedStep(_loss_inputs(b), theta, lambda: None, lambda: None)
    pageable = [t.cpu() for t in _loss_inputs(b)]
    with pytest.raises(ValueError, match="page-locked"):
        pipe.step(pageable, theta.cpu().pin_memory())
    with pytest.raises(ValueError, match="one host tensor"):
        pipe.step(pageable[:2], theta.cpu().pin_memory())
