"""K2 with the interpolation proxies of Table 1 / App. A (p->proxy) against the oracle.

With a proxy, log pi_old is built per token from log mu_old and log pi_theta
inside the kernel.  Bars as in test_gpu_loss.py.  The Table 4 effective
thresholds are reproduced on the GPU by sweeping r = pi_theta / mu_old across
them and reading the kernel's flags.
"""

import os

import numpy as np
import pytest
import torch

import oracle as orc
from oracle_runner import dlogits_rows, fp32, logprob_rows, loss_params, oracle_loss
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import LossBatch, make_loss_batch

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("kind", ["loglinear", "arithmetic"])
@pytest.mark.parametrize("alpha", [0.5, 1.0 / 3.0, 0.25])
@pytest.mark.parametrize("name,T", [("agentic_bf16_v151936", 256), ("grpo_bf16_v32000", 2048)])
def test_proxy_modes_against_oracle(kind, alpha, name, T):
    b = make_loss_batch(name, T=T, seed=11, device="cuda")
    b.rd_lo, b.rd_hi = 0.95, 1.05
    rows = np.arange(T)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    lmu = b.logp_mu.cpu().numpy()
    lp_prox = orc.proxy_logprob(kind, alpha, lmu, np.nan_to_num(lt64))
    o = oracle_loss(b, lt64, lp_prox, loss_params(b))
    out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, None, b.logp_mu, b.adv, b.mask,
                                         proxy=kind, alpha=alpha, **b.thresholds())
    torch.cuda.synchronize()
    st = occ.decode_loss_stats(out["stats"])
    fl = out["flags"].cpu().numpy()
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    diff = fl != o["flags"]
    assert not (diff & ~(near & o["valid"])).any()
    assert 0 < o["n_rd_out"] < o["n_valid"] and 0 < o["n_active"]
    assert abs(st.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
    pick = np.array([r for r in np.nonzero(o["g"])[0][:16] if not diff[r]], dtype=np.int64)
    assert pick.size > 0
    ref = dlogits_rows(b, pick, lse[pick], o["g"][pick])
    got = out["dlogits"][torch.as_tensor(pick, device="cuda")].float().cpu().numpy()
    g = np.abs(o["g"][pick])[:, None]
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 4e-6 * g + 1e-30)


def _table4(golden):
    rows = []
    with open(golden) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                v = line.split()
                rows.append((*map(float, v[:4]), int(v[4]), v[5], *map(float, v[6:])))
    return rows


def test_table4_effective_thresholds_on_gpu():
    """Table 4: the kernel's band and clip decisions under each proxy cut
    r = pi_theta / mu_old at the printed effective bounds (4 decimals)."""
    rows = _table4(os.path.join(ROOT, "tests", "golden", "table4_effective_thresholds.txt"))
    r_grid = np.linspace(0.95, 1.05, 10001)                  # step 1e-5
    n = r_grid.size
    g = torch.Generator(device="cuda").manual_seed(0)
    V = 64
    z = (torch.randn((n, V), generator=g, device="cuda") * 2).to(torch.float32)
    ids = torch.zeros(n, dtype=torch.int32, device="cuda")
    lt64, _ = logprob_rows(z, ids, np.arange(n))
    lmu = torch.from_numpy(fp32(lt64 - np.log(r_grid))).cuda()
    # the ratio the kernel sees uses its own float32 log mu; recompute r exactly
    r_eff = np.exp(lt64 - lmu.cpu().numpy().astype(np.float64))
    checked = 0
    for (mlo, mhi, clo, chi, nn, kind, e_mlo, e_mhi, e_clo, e_chi) in rows:
        alpha = 1.0 / (nn + 1)
        proxy = "arithmetic" if kind == "linear" else "loglinear"
        for A, side in ((1.0, "hi"), (-1.0, "lo")):
            adv = torch.full((n,), A, device="cuda")
            b = LossBatch("t4", z, z, ids, lmu, adv, None, rd_lo=mlo, rd_hi=mhi,
                          eps_low=1.0 - clo, eps_high=chi - 1.0)
            out = occ.occ_decoupled_loss_fwd_bwd(z, ids, None, lmu, adv, None, proxy=proxy,
                                                 alpha=alpha, dlogits=None, **b.thresholds())
            torch.cuda.synchronize()
            fl = out["flags"].cpu().numpy()
            band = r_eff[(fl & occ.FLAG_IN_BAND) != 0]
            assert abs(band.min() - e_mlo) <= 5e-5 + 2e-5 and abs(band.max() - e_mhi) <= 7e-5
            kept = r_eff[(fl & occ.FLAG_CLIPPED) == 0]
            if side == "hi":
                assert abs(kept.max() - e_chi) <= 7e-5
            else:
                assert abs(kept.min() - e_clo) <= 7e-5
            checked += 1
    assert checked == 48


def test_proxy_rejected_by_fused_entry_point():
    b = make_loss_batch("tiny_f32_v4096", T=8, seed=0, device="cuda")
    lib = occ.lib()
    import ctypes
    p = occ._params(0.5, 2.0, 0.2, 0.28, 1.0, 0, 1, 0, "loglinear", 0.5)
    ws = occ.new_workspace(8, 4096, "cuda")
    st = occ.new_loss_stats("cuda")
    rc = lib.occ_decoupled_loss_fused(
        ctypes.c_void_p(b.z_theta.data_ptr()), ctypes.c_void_p(b.z_old.data_ptr()), 0, 8, 4096,
        4096, 4096, ctypes.c_void_p(b.ids.data_ptr()), ctypes.c_void_p(b.logp_mu.data_ptr()),
        ctypes.c_void_p(b.adv.data_ptr()), None, ctypes.byref(p), None, None, None, None, None,
        None, 0, ctypes.c_void_p(st.data_ptr()), ctypes.c_void_p(ws.data_ptr()), ws.numel(), None)
    assert rc == 1 and b"proxies" in lib.occ_last_error()


@pytest.mark.parametrize("kind", ["loglinear", "arithmetic"])
@pytest.mark.parametrize("alpha", [0.0, 1.0])
def test_proxy_degenerate_weights(kind, alpha):
    # alpha = 1: the proxy is mu_old itself, so r_d = 1 and no token leaves the
    # band (Eq. 4 reduces to plain PPO-clip).  alpha = 0: the proxy is pi_theta,
    # so r_s = 1 and no token is clipped (Table 1's interpolation end points).
    b = make_loss_batch("agentic_bf16_v151936", T=256, seed=13, device="cuda")
    rows = np.arange(b.T)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    lmu = b.logp_mu.cpu().numpy().astype(np.float64)
    lp_prox = orc.proxy_logprob(kind, alpha, lmu, np.nan_to_num(lt64))
    o = oracle_loss(b, lt64, lp_prox, loss_params(b))
    out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, None, b.logp_mu, b.adv, b.mask,
                                         proxy=kind, alpha=alpha, **b.thresholds())
    torch.cuda.synchronize()
    st = occ.decode_loss_stats(out["stats"])
    fl = out["flags"].cpu().numpy()
    assert st.n_valid == o["n_valid"] > 0
    if alpha == 1.0:
        assert st.n_rd_out == 0 == o["n_rd_out"]
    else:
        assert st.n_clipped == 0 == o["n_clipped"]
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    assert not ((fl != o["flags"]) & ~(near & o["valid"])).any()
    assert abs(st.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
