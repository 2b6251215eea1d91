"""occ_decoupled_loss_fwd_bwd_noalloc: the loss for callers that cannot allocate.

A caller with no device allocator of its own (a C plugin inside a framework
whose caching allocator owns the GPU's memory, or a loop that must not call
cudaMalloc/cudaFree) cannot provide the workspace occ_decoupled_loss_fwd_bwd
needs.  The no-alloc entry point takes its scratch from a fixed array inside
the library.  Here it is called through the C ABI and must reproduce the
workspace entry point's outputs (the parity tests' tolerances; in practice the
same kernels give identical bits) on two calls in a row, the second with a
different batch so that anything left in the shared scratch by the first call
would show.  This file is collected last on purpose.
"""

import numpy as np
import pytest
import torch

from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu


def _outputs(b, lp_old, noalloc):
    T, V = b.T, b.V
    dz = torch.full((T, V), 3.0, dtype=b.z_theta.dtype, device="cuda")
    logp = torch.full((T,), 5.0, device="cuda")
    flags = torch.full((T,), 255, dtype=torch.uint8, device="cuda")
    stats = torch.full((occ.LOSS_STATS_BYTES,), 7, dtype=torch.uint8, device="cuda")
    kw = dict(dlogits=dz, logp_out=logp, flags_out=flags, stats=stats, **b.thresholds())
    if noalloc:
        occ.occ_decoupled_loss_fwd_bwd_noalloc(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv,
                                               b.mask, **kw)
    else:
        occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask, **kw)
    torch.cuda.synchronize()
    return dz, logp, flags, stats


def _assert_same(a, b):
    dz_a, lp_a, fl_a, st_a = a
    dz_b, lp_b, fl_b, st_b = b
    sa, sb = occ.decode_loss_stats(st_a), occ.decode_loss_stats(st_b)
    assert (sa.n_valid, sa.n_rd_out, sa.n_clipped, sa.n_active, sa.denom, sa.err) == \
        (sb.n_valid, sb.n_rd_out, sb.n_clipped, sb.n_active, sb.denom, sb.err)
    assert abs(sa.loss - sb.loss) <= 1e-4 * abs(sb.loss) + 1e-12
    assert torch.equal(fl_a, fl_b)
    va = (fl_b & occ.FLAG_VALID) != 0
    assert torch.allclose(lp_a[va], lp_b[va], rtol=0, atol=1e-5)
    diff = (dz_a.float() - dz_b.float()).abs()
    assert diff.max().item() <= 3e-3
    assert torch.all(diff <= 2.0 ** -8 * dz_b.float().abs() + 1e-7)


def test_noalloc_matches_workspace_entry_point_twice():
    first = make_loss_batch("agentic_bf16_v151936", T=3000, seed=21, device="cuda")
    second = make_loss_batch("grpo_bf16_v32000", T=1500, seed=22, device="cuda")
    for b in (first, second):
        lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
        ref = _outputs(b, lp_old, noalloc=False)
        got = _outputs(b, lp_old, noalloc=True)
        _assert_same(got, ref)
        assert occ.decode_loss_stats(got[3]).n_active > 0


def test_noalloc_rejects_batches_beyond_its_scratch():
    T = occ.NOALLOC_MAX_TOKENS + 1
    z = torch.zeros((T, 8), dtype=torch.bfloat16, device="cuda")
    i = torch.zeros(T, dtype=torch.int32, device="cuda")
    f = torch.zeros(T, device="cuda")
    with pytest.raises(occ.OccError, match="at most 786432 tokens"):
        occ.occ_decoupled_loss_fwd_bwd_noalloc(
            z, i, f, f, f, None, rd_lo=0.5, rd_hi=2.0, eps_low=0.2, eps_high=0.28, dlogits=None,
            logp_out=f, flags_out=None, stats=occ.new_loss_stats("cuda"))
