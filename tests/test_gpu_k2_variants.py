"""The K2 launch shapes that the options select, against the oracle.

K2 picks its CTA size, shared-memory head and loads in flight by row size;
the options k2_threads, k2_head_bytes and k2_unroll override that choice for
measurements.  Every shape must give the same results: each runs here on a
long-row batch (V = 151936) and a short-row one (V = 32000), bf16 and float32
gradients, against the oracle.
"""

import numpy as np
import pytest
import torch

from oracle_runner import dlogits_rows, fp32, logprob_rows, loss_params, oracle_loss
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu

SHAPES = [dict(k2_threads=128), dict(k2_threads=256), dict(k2_threads=512, k2_unroll=4),
          dict(k2_threads=512, k2_head_bytes=0), dict(k2_threads=256, k2_head_bytes=32768)]


@pytest.mark.parametrize("shape", SHAPES, ids=lambda d: ",".join(f"{k}={v}" for k, v in d.items()))
@pytest.mark.parametrize("name,T,f32", [("agentic_bf16_v151936", 200, False),
                                        ("grpo_bf16_v32000", 300, True)])
def test_k2_launch_shape_against_oracle(shape, name, T, f32):
    b = make_loss_batch(name, T=T, seed=7, device="cuda")
    rows = np.arange(b.T)
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    o = oracle_loss(b, lt64, fp32(lo64), loss_params(b))
    with occ.options(**shape):
        out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, torch.from_numpy(fp32(lo64)).cuda(),
                                             b.logp_mu, b.adv, b.mask, dlogits_f32=f32,
                                             **b.thresholds())
        assert occ.occ_last_kernel() == "k2_loss_l2"
    torch.cuda.synchronize()
    s = occ.decode_loss_stats(out["stats"])
    fl = out["flags"].cpu().numpy()
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    assert not ((fl != o["flags"]) & ~near).any()
    assert abs(s.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
    v = o["valid"]
    assert np.abs(out["logp"].cpu().numpy()[v] - lt64[v]).max() <= 1e-5
    pick = np.unique(np.concatenate([np.nonzero(o["g"])[0][:12], [0, b.T - 1]]))
    ref = dlogits_rows(b, pick, lse[pick], o["g"][pick])
    got = out["dlogits"][torch.as_tensor(pick, device="cuda")].float().cpu().numpy()
    g = np.abs(o["g"][pick])[:, None]
    rel = 2e-6 if f32 else 2.0 ** -8
    assert np.all(np.abs(got - ref) <= rel * np.abs(ref) + 4e-6 * g + 1e-30)


@pytest.mark.parametrize("unroll", [None, 4, 6, 8])
def test_k2_peeled_long_rows_every_unroll(unroll):
    """Long rows off a 16-byte boundary (V = 151937 bf16, odd row stride) run
    the peeled 512-thread kernel; each number of vectors in flight gives the
    oracle's results on every token."""
    T, V = 24, 151937
    g = torch.Generator(device="cuda").manual_seed(11)
    z = (torch.randn((T, V), generator=g, device="cuda") * 2.5).to(torch.bfloat16)
    zo = (z.float() + 0.3 * torch.randn((T, V), generator=g, device="cuda")).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    ids[0], ids[-1] = 0, V - 1
    rows = np.arange(T)
    lo64, _ = logprob_rows(zo, ids, rows)
    lt64, lse = logprob_rows(z, ids, rows)
    from paper_2605_12070_gb300.workloads import LossBatch
    b = LossBatch(name="peeled", z_theta=z, z_old=zo, ids=ids,
                  logp_mu=torch.from_numpy(fp32(lo64 + np.random.default_rng(11).normal(0, 0.3, T))).cuda(),
                  adv=torch.randn(T, generator=g, device="cuda"),
                  mask=(torch.rand(T, generator=g, device="cuda") < 0.8).to(torch.uint8),
                  rd_lo=0.7, rd_hi=1.4, eps_low=0.2, eps_high=0.28)
    assert z.stride(0) % 2 == 1
    o = oracle_loss(b, lt64, fp32(lo64), loss_params(b))
    shape = {} if unroll is None else dict(k2_threads=512, k2_unroll=unroll)
    with occ.options(**shape):
        out = occ.occ_decoupled_loss_fwd_bwd(z, ids, torch.from_numpy(fp32(lo64)).cuda(), b.logp_mu,
                                             b.adv, b.mask, **b.thresholds())
        # the automatic shape keeps 128 KB of each row in tensor memory; a shape option the plain kernel
        assert occ.occ_last_kernel() == ("k2_loss_l2/peel/tmem" if unroll is None else "k2_loss_l2/peel")
    torch.cuda.synchronize()
    s = occ.decode_loss_stats(out["stats"])
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    assert not ((out["flags"].cpu().numpy() != o["flags"]) & ~near).any()
    assert abs(s.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
    v = o["valid"]
    assert np.abs(out["logp"].cpu().numpy()[v] - lt64[v]).max() <= 1e-5
    ref = dlogits_rows(b, rows, lse, o["g"])
    got = out["dlogits"].float().cpu().numpy()
    g_ = np.abs(o["g"])[:, None]
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 4e-6 * g_ + 1e-30)
