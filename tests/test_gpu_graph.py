"""The training step replays from a CUDA graph.

The loss entry points and the EWMA update allocate nothing, never synchronise
and keep their cross-step state (the token count N, the loss statistics, the
EWMA weight w and the low-ratio streak) in device memory, so a captured step
(K0, the loss kernel(s), the finalize, the EWMA prologue and body) replays
without the host.  The kernels are deterministic: every replay must give the
bits of the same eager call sequence, including the EWMA state that advances
from step to step (App. B recursion and the Sec. 5.2 reset rule).
"""

import pytest
import torch

from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_ewma_buffers, make_loss_batch

pytestmark = pytest.mark.gpu

STEPS = 3


def _buffers(b, n_params):
    T, V = b.T, b.V
    dev = "cuda"
    return {
        "dlogits": torch.empty((T, V), dtype=torch.bfloat16, device=dev),
        "logp": torch.empty(T, dtype=torch.float32, device=dev),
        "lp_old": torch.empty(T, dtype=torch.float32, device=dev),
        "flags": torch.empty(T, dtype=torch.uint8, device=dev),
        "stats": occ.new_loss_stats(dev),
        "ws": occ.new_workspace(T, V, dev),
    }


def _step(path, b, o, theta, theta_prox, state, tau):
    if path == "fused":
        occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                     **b.thresholds(), dlogits=o["dlogits"], logp_out=o["logp"],
                                     logp_old_out=o["lp_old"], flags_out=o["flags"],
                                     stats=o["stats"], workspace=o["ws"])
    else:
        occ.occ_token_logprob(b.z_old, b.ids, logp_out=o["lp_old"])
        occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, o["lp_old"], b.logp_mu, b.adv, b.mask,
                                       **b.thresholds(), dlogits=o["dlogits"],
                                       logp_out=o["logp"], flags_out=o["flags"],
                                       stats=o["stats"], workspace=o["ws"])
    occ.occ_ewma_update(theta_prox, theta, 0.75, state, stats=o["stats"], tau=tau)


@pytest.mark.parametrize("path", ["fused", "two-call"])
@pytest.mark.parametrize("tau", [0.5, 0.95])  # 0.95 > rho: every step resets
def test_captured_step_replays_bit_identically(path, tau):
    b = make_loss_batch("agentic_bf16_v151936", T=384, seed=21, device="cuda")
    theta, theta_prox0 = make_ewma_buffers(1_000_003, seed=21, device="cuda")
    state0 = occ.new_ewma_state("cuda", w0=2.0)

    eager = _buffers(b, theta.numel())
    tp_e, st_e = theta_prox0.clone(), state0.clone()
    for _ in range(STEPS):
        _step(path, b, eager, theta, tp_e, st_e, tau)
    torch.cuda.synchronize()

    graphed = _buffers(b, theta.numel())
    tp_g, st_g = theta_prox0.clone(), state0.clone()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        _step(path, b, graphed, theta, tp_g, st_g, tau)
    # capture records the launches without running them
    torch.cuda.synchronize()
    assert torch.equal(tp_g, theta_prox0) and torch.equal(st_g, state0)
    for _ in range(STEPS):
        g.replay()
    torch.cuda.synchronize()

    for k in ("dlogits", "logp", "lp_old", "flags", "stats"):
        assert torch.equal(graphed[k], eager[k]), k
    assert torch.equal(tp_g, tp_e)
    assert torch.equal(st_g, st_e)
    st = occ.decode_ewma_state(st_g)
    assert st.n_resets == (STEPS if tau > occ.decode_loss_stats(eager["stats"]).rho else 0)
