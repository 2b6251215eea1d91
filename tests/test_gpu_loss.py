"""K0 + K2 parity: occ_decoupled_loss_fwd_bwd against the float64 oracle (R1..R9).

Parity bars: mask and clip flags bit-exact except tokens whose oracle
log-ratio lies within 1e-6 of the deciding threshold; log-probabilities within
2e-3 absolute (tight bound 1e-5); loss within 1e-4 relative; dlogits within
3e-3 absolute.  The dlogits bound used here is tighter and derived from the
output rounding: |err| <= 2^-8 |ref| + 4e-6 |g_t| for bf16 output and
<= 2e-6 |ref| + 4e-6 |g_t| for float32 output (g_t = the row's gradient scale).
"""

import numpy as np
import pytest
import torch

from oracle import FLAG_ACTIVE, FLAG_CLIPPED, FLAG_IN_BAND
from kernel_choice import expected_kernel
from oracle_runner import dlogits_rows, fp32, logprob_rows, loss_params, oracle_loss
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu

EXEMPT = 1e-6
LOGP_TOL, LOGP_TIGHT = 2e-3, 1e-5
LOSS_RTOL = 1e-4
DZ_ABS = 3e-3


def _compare(batch, out, o, lp_theta64, exempt_extra=None, dz_rows=None, lse=None,
             out_f32=False):
    """Checks GPU outputs against the oracle dict ``o`` (all tokens)."""
    st = occ.decode_loss_stats(out["stats"])
    valid = o["valid"]
    assert st.denom == o["N"] and st.n_valid == o["n_valid"]
    # log-probabilities of valid tokens
    glp = out["logp"].cpu().numpy().astype(np.float64)
    if valid.any():
        err = np.abs(glp[valid] - lp_theta64[valid])
        assert err.max() <= LOGP_TOL and err.max() <= LOGP_TIGHT, f"max |dlogp| {err.max():.3g}"
    assert np.all(glp[~valid & np.isfinite(glp)] == 0.0)
    # flags: bit-exact except near-threshold tokens
    gfl = out["flags"].cpu().numpy()
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= EXEMPT
    if exempt_extra is not None:
        near |= exempt_extra
    diff = gfl != o["flags"]
    bad = diff & ~(near & valid)
    assert not bad.any(), (f"{bad.sum()} non-exempt flag mismatches, e.g. t={np.nonzero(bad)[0][:5]} "
                           f"gpu={gfl[bad][:5]} ref={o['flags'][bad][:5]}")
    nflip = int(diff.sum())
    for key, bit, inv in (("n_rd_out", FLAG_IN_BAND, True), ("n_clipped", FLAG_CLIPPED, False),
                          ("n_active", FLAG_ACTIVE, False)):
        assert abs(getattr(st, key) - o[key]) <= nflip, key
    if nflip == 0:
        assert (st.n_rd_out, st.n_clipped, st.n_active) == (o["n_rd_out"], o["n_clipped"],
                                                            o["n_active"])
    # loss: band flips move the loss by at most |w_d s_t| / N each
    slack = 0.0
    if nflip and o["N"]:
        flipped_band = diff & (((gfl ^ o["flags"]) & FLAG_IN_BAND) != 0)
        w = np.maximum(o["r_d"], 1.0)
        slack = float(np.sum(np.abs(w * o["r_s"] * batch.adv.cpu().numpy())[flipped_band])) / o["N"]
    assert abs(st.loss - o["loss"]) <= LOSS_RTOL * abs(o["loss"]) + slack + 1e-12, \
        (st.loss, o["loss"])
    assert st.err == 0
    # dlogits on the requested rows (flag-flipped rows skipped)
    if dz_rows is not None and out["dlogits"] is not None:
        rows = np.array([r for r in dz_rows if not diff[r]], dtype=np.int64)
        ref = dlogits_rows(batch, rows, lse, o["g"][rows])
        got = out["dlogits"][torch.as_tensor(rows, device="cuda")].float().cpu().numpy()
        g = np.abs(o["g"][rows])[:, None]
        tol = (2e-6 * np.abs(ref) if out_f32 else 2.0 ** -8 * np.abs(ref)) + 4e-6 * g
        err = np.abs(got - ref)
        assert err.max() <= DZ_ABS
        assert np.all(err <= tol + 1e-30), f"dz err {(err - tol).max():.3g}"
        # rows that carry no gradient are exactly zero
        dead = o["g"][rows] == 0.0
        assert np.all(got[dead] == 0.0)
    return st


def _run(batch, lp_old32, dz="new", **kw):
    lp_old = torch.from_numpy(lp_old32).to("cuda")
    out = occ.occ_decoupled_loss_fwd_bwd(batch.z_theta, batch.ids, lp_old, batch.logp_mu,
                                         batch.adv, batch.mask, dlogits=dz,
                                         **batch.thresholds(), **kw)
    torch.cuda.synchronize()
    return out


def _full_parity(batch, rd_weight=1, dlogits_f32=False, grad_scale=1.0, n_dz_rows=24, seed=0):
    T = batch.T
    rows = np.arange(T)
    lp_old64, _ = logprob_rows(batch.z_old, batch.ids, rows)
    lp_th64, lse_th = logprob_rows(batch.z_theta, batch.ids, rows)
    lp_old32 = fp32(lp_old64)
    p = loss_params(batch, rd_weight=rd_weight, grad_scale=grad_scale)
    o = oracle_loss(batch, lp_th64, lp_old32, p)
    out = _run(batch, lp_old32, rd_weight=rd_weight, grad_scale=grad_scale,
               dlogits_f32=dlogits_f32)
    rng = np.random.default_rng(seed)
    act = np.nonzero(o["g"] != 0)[0]
    pick = [0, T - 1]
    if act.size:
        pick += list(rng.choice(act, size=min(n_dz_rows, act.size), replace=False))
    pick += list(rng.choice(T, size=min(8, T), replace=False))
    dz_rows = np.unique(np.array(pick))
    if o["n_valid"] > 0:  # the batch must exercise the gradient, not compare zeros
        assert np.count_nonzero(o["g"][dz_rows]) > 0, "no compared row carries a gradient"
    return _compare(batch, out, o, lp_th64, dz_rows=dz_rows, lse=lse_th[dz_rows],
                    out_f32=dlogits_f32 or batch.z_theta.dtype == torch.float32), o


@pytest.mark.parametrize("rd_weight", [1, 0])
def test_tiny_f32_full(rd_weight):
    b = make_loss_batch("tiny_f32_v4096", seed=0, device="cuda")
    st, o = _full_parity(b, rd_weight=rd_weight)
    assert o["n_active"] > 0


@pytest.mark.parametrize("name,T", [("grpo_bf16_v32000", 700), ("agentic_bf16_v151936", 300),
                                    ("heavytail_bf16_v151936", 300)])
@pytest.mark.parametrize("dlogits_f32", [False, True])
def test_workloads_reduced(name, T, dlogits_f32):
    b = make_loss_batch(name, T=T, seed=2, device="cuda")
    _full_parity(b, dlogits_f32=dlogits_f32)


def test_grad_scale_makes_dz_order_one():
    # grad_scale = N turns dlogits into r A (1[v=y] - p): O(1) values, so the
    # 3e-3 absolute bound is a meaningful check.
    b = make_loss_batch("agentic_bf16_v151936", T=256, seed=3, device="cuda")
    N = int(b.mask.sum().item())
    _full_parity(b, grad_scale=float(N), dlogits_f32=True)


def test_grpo_full_size():
    b = make_loss_batch("grpo_bf16_v32000", seed=0, device="cuda")
    st, o = _full_parity(b, n_dz_rows=48)
    assert 0 < st.n_clipped < st.n_valid


def test_heavytail_full_size_counts_exact():
    b = make_loss_batch("heavytail_bf16_v151936", seed=0, device="cuda")
    st, o = _full_parity(b, n_dz_rows=32)
    frac = o["n_rd_out"] / o["n_valid"]
    assert 0.01 <= frac <= 0.05, frac       # the workload's stated 1-5% outside the band
    assert (st.n_rd_out, st.n_clipped, st.n_active) == (o["n_rd_out"], o["n_clipped"],
                                                        o["n_active"])


# ------------------------------------------------------------------ edge cases

def _edge_batch(T, V, dtype, seed, mask_p=0.8, ld=None, offset=0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    ldv = V if ld is None else ld
    buf = (torch.randn((T, ldv + offset), generator=g, device="cuda") * 2.5).to(dtype)
    z = buf[:, offset:offset + V]
    zo = (z.float() + 0.3 * torch.randn((T, V), generator=g, device="cuda")).to(dtype)
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    if T:
        ids[0] = 0
        ids[-1] = V - 1
    adv = torch.randn(T, generator=g, device="cuda")
    mask = (torch.rand(T, generator=g, device="cuda") < mask_p).to(torch.uint8)
    from paper_2605_12070_gb300.workloads import LossBatch
    b = LossBatch(name="edge", z_theta=z, z_old=zo, ids=ids, logp_mu=None, adv=adv, mask=mask,
                  rd_lo=0.7, rd_hi=1.4, eps_low=0.2, eps_high=0.28)
    lp_old64, _ = logprob_rows(zo, ids, np.arange(T))
    b.logp_mu = torch.from_numpy(fp32(lp_old64 + np.random.default_rng(seed).normal(0, 0.3, T))).to("cuda")
    return b, lp_old64


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [1, 7, 8, 9, 63, 65, 127, 129, 4095, 4097, 8184, 8192, 8200, 16376,
                               16384, 16392, 20000, 50000, 65536, 65536 + 3, 65544])
def test_vocab_edges(V, dtype):
    # besides the ragged and tiny rows: rows of one vector less, exactly and
    # one vector more than whole rounds of loads (forward and re-read, 128- and
    # 512-thread tiers), where the last partial round of a row is empty or
    # holds a single vector
    T = 37
    b, lp_old64 = _edge_batch(T, V, dtype, seed=V)
    lp_th64, lse = logprob_rows(b.z_theta, b.ids, np.arange(T))
    p = loss_params(b)
    o = oracle_loss(b, lp_th64, fp32(lp_old64), p)
    out = _run(b, fp32(lp_old64))
    assert occ.occ_last_kernel() == expected_kernel("k2", V, b.z_theta.element_size())
    _compare(b, out, o, lp_th64, dz_rows=np.arange(T), lse=lse,
             out_f32=dtype == torch.float32)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("layout", ["ld_pad", "offset", "ld_odd"])
def test_strided_and_misaligned(dtype, layout):
    T, V = 23, 3001
    kw = dict(ld_pad=dict(ld=3008), offset=dict(ld=3010, offset=1), ld_odd=dict(ld=3003))[layout]
    b, lp_old64 = _edge_batch(T, V, dtype, seed=5, **kw)
    lp_th64, lse = logprob_rows(b.z_theta, b.ids, np.arange(T))
    o = oracle_loss(b, lp_th64, fp32(lp_old64), loss_params(b))
    # dlogits into a padded buffer of its own stride
    dz_buf = torch.full((T, V + 7), 7.0, dtype=dtype, device="cuda")
    out = _run(b, fp32(lp_old64), dz=dz_buf[:, :V])
    # gradient rows at other byte offsets than the logits rows: element loads
    assert occ.occ_last_kernel() == ("k2_loss_l2" if layout == "ld_pad" else "k2_loss_stream")
    out["dlogits"] = dz_buf[:, :V]
    _compare(b, out, o, lp_th64, dz_rows=np.arange(T), lse=lse, out_f32=dtype == torch.float32)
    assert torch.all(dz_buf[:, V:] == 7.0)   # padding untouched


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [3001, 20003])
def test_misaligned_rows_with_matching_gradient_layout(dtype, V):
    """Rows off a 16-byte boundary whose gradient rows have the same byte
    offsets (a buffer of the same stride and offset, in place, or no gradient)
    run the peeled vector kernel.  The odd row stride gives every row-start
    residue; the sampled token of row 0 lies in its scalar prefix and that of
    the last row in its scalar tail."""
    T, off = 29, 1
    b, lp_old64 = _edge_batch(T, V, dtype, seed=V + 1, ld=V + 1, offset=off)
    peeled = expected_kernel("k2", V, b.z_theta.element_size())  # "/tmem": the f32 rows
    assert peeled.startswith("k2_loss_l2/peel")
    stride = b.z_theta.stride(0)
    assert stride % 2 == 1 and b.z_theta.data_ptr() % 16 != 0
    lp_th64, lse = logprob_rows(b.z_theta, b.ids, np.arange(T))
    o = oracle_loss(b, lp_th64, fp32(lp_old64), loss_params(b))
    dz_buf = torch.full((T, stride), 7.0, dtype=dtype, device="cuda")
    dz = dz_buf[:, off:off + V]
    out = _run(b, fp32(lp_old64), dz=dz)
    assert occ.occ_last_kernel() == peeled
    out["dlogits"] = dz
    _compare(b, out, o, lp_th64, dz_rows=np.arange(T), lse=lse, out_f32=dtype == torch.float32)
    assert torch.all(dz_buf[:, :off] == 7.0) and torch.all(dz_buf[:, off + V:] == 7.0)
    # in place over a copy with the same layout: the same kernel, the same bits
    buf2 = torch.empty((T, stride), dtype=dtype, device="cuda")
    z2 = buf2[:, off:off + V]
    z2.copy_(b.z_theta)
    lp_old = torch.from_numpy(fp32(lp_old64)).to("cuda")
    out2 = occ.occ_decoupled_loss_fwd_bwd(z2, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                          dlogits="inplace", **b.thresholds())
    assert occ.occ_last_kernel() == peeled
    # forward only
    out3 = _run(b, fp32(lp_old64), dz=None)
    assert occ.occ_last_kernel() == peeled
    assert torch.equal(z2, dz) and torch.equal(out2["stats"], out["stats"])
    assert torch.equal(out3["stats"], out["stats"]) and torch.equal(out3["logp"], out["logp"])


@pytest.mark.parametrize("V", [600_000, 900_001])
def test_large_vocab_paths(V):
    # 600k bf16 rows need an 8-CTA cluster; 900k exceed it and take the
    # streaming kernel.
    T = 6
    b, lp_old64 = _edge_batch(T, V, torch.bfloat16, seed=11, mask_p=1.0)
    lp_th64, lse = logprob_rows(b.z_theta, b.ids, np.arange(T))
    o = oracle_loss(b, lp_th64, fp32(lp_old64), loss_params(b))
    out = _run(b, fp32(lp_old64))
    _compare(b, out, o, lp_th64, dz_rows=np.arange(T), lse=lse)


def test_in_place_dlogits_matches_out_of_place():
    b, lp_old64 = _edge_batch(64, 32000, torch.bfloat16, seed=3)
    ref = _run(b, fp32(lp_old64))
    z2 = b.z_theta.clone()
    lp_old = torch.from_numpy(fp32(lp_old64)).to("cuda")
    out = occ.occ_decoupled_loss_fwd_bwd(z2, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                         dlogits="inplace", **b.thresholds())
    torch.cuda.synchronize()
    assert out["dlogits"].data_ptr() == z2.data_ptr()
    assert torch.equal(z2, ref["dlogits"])
    assert torch.equal(out["stats"], ref["stats"]) and torch.equal(out["flags"], ref["flags"])


def test_bad_ids_all_masked_zero_adv_and_empty():
    b, lp_old64 = _edge_batch(16, 1000, torch.float32, seed=9, mask_p=1.0)
    b.ids[3] = -5
    b.ids[7] = 1000
    b.adv[5] = 0.0
    out = _run(b, fp32(np.nan_to_num(lp_old64)))
    st = occ.decode_loss_stats(out["stats"])
    assert st.err == occ.DATA_ERR_BAD_ID
    assert st.n_valid == 14 and st.denom == 14
    lp = out["logp"].cpu().numpy()
    assert np.isnan(lp[3]) and np.isnan(lp[7])
    fl = out["flags"].cpu().numpy()
    assert fl[3] == 0 and fl[7] == 0
    dz = out["dlogits"].cpu()
    assert torch.all(dz[3] == 0) and torch.all(dz[7] == 0) and torch.all(dz[5] == 0)
    # everything masked: loss 0, N 0, all-zero gradient
    b.mask.zero_()
    out = _run(b, fp32(np.nan_to_num(lp_old64)))
    st = occ.decode_loss_stats(out["stats"])
    assert (st.loss, st.loss_sum, st.denom, st.n_valid) == (0.0, 0.0, 0, 0)
    assert torch.all(out["dlogits"] == 0)
    # T = 0
    e = torch.empty((0, 1000), device="cuda")
    z0 = torch.empty(0, device="cuda")
    i0 = torch.empty(0, dtype=torch.int32, device="cuda")
    out = occ.occ_decoupled_loss_fwd_bwd(e, i0, z0, z0, z0, None, rd_lo=0.5, rd_hi=2, eps_low=0.2,
                                         eps_high=0.28)
    st = occ.decode_loss_stats(out["stats"])
    assert (st.loss, st.denom, st.n_valid) == (0.0, 0, 0)


def test_denominator_and_forward_only():
    b, lp_old64 = _edge_batch(50, 2048, torch.bfloat16, seed=4)
    full = _run(b, fp32(lp_old64))
    fwd = _run(b, fp32(lp_old64), dz=None, denom=200, grad_scale=3.0)
    s1 = occ.decode_loss_stats(full["stats"])
    s2 = occ.decode_loss_stats(fwd["stats"])
    assert fwd["dlogits"] is None and s2.denom == 200
    assert abs(s2.loss * 200 - s1.loss * s1.denom) <= 1e-12 + 1e-7 * abs(s1.loss_sum)
    assert torch.equal(full["flags"], fwd["flags"]) and torch.equal(full["logp"], fwd["logp"])


def test_deterministic_repeat():
    b = make_loss_batch("agentic_bf16_v151936", T=512, seed=5, device="cuda")
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    a = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                       **b.thresholds())
    c = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                       **b.thresholds())
    torch.cuda.synchronize()
    assert torch.equal(a["stats"], c["stats"]) and torch.equal(a["dlogits"], c["dlogits"])


def test_invalid_arguments_raise_before_launch():
    z = torch.zeros((4, 16), device="cuda")
    i = torch.zeros(4, dtype=torch.int32, device="cuda")
    f = torch.zeros(4, device="cuda")
    with pytest.raises(occ.OccError, match="invalid argument"):
        occ.occ_decoupled_loss_fwd_bwd(z, i, f, f, f, None, rd_lo=2.0, rd_hi=0.5, eps_low=0.2,
                                       eps_high=0.28)
    with pytest.raises(occ.OccError, match="workspace"):
        occ.occ_decoupled_loss_fwd_bwd(z, i, f, f, f, None, rd_lo=0.5, rd_hi=2, eps_low=0.2,
                                       eps_high=0.28,
                                       workspace=torch.empty(8, dtype=torch.uint8, device="cuda"))
    with pytest.raises(occ.OccError, match="overlaps"):
        big = torch.zeros((5, 16), device="cuda")
        occ.occ_decoupled_loss_fwd_bwd(big[:4], i, f, f, f, None, rd_lo=0.5, rd_hi=2, eps_low=0.2,
                                       eps_high=0.28, dlogits=big[1:5])


@pytest.mark.parametrize("rd_weight", [1, 0])
def test_open_band_roles_of_table5(rd_weight):
    # Table 5's "PPO-EWMA" and "linear_prox" rows weight by r_2 without masking
    # it (r_2 * M(r_1)): an open band [0, inf) keeps every token in band.  With
    # rd_weight = 0 the same band gives plain M(r_1) on pi_old.  The heavy-tailed
    # batch puts many tokens far outside any finite band, so r_d reaches the
    # gradient with large weights.
    b = make_loss_batch("heavytail_bf16_v151936", T=300, seed=3, device="cuda")
    b.rd_lo, b.rd_hi = 0.0, float("inf")
    st, o = _full_parity(b, rd_weight=rd_weight)
    assert st.n_rd_out == 0 == o["n_rd_out"]
    v = o["valid"]
    assert np.all((o["flags"][v] & FLAG_IN_BAND) != 0)
    if rd_weight:
        assert np.max(o["r_d"][v]) > 2.0 or np.min(o["r_d"][v]) < 0.5  # weights far from 1


@pytest.mark.parametrize("rd_weight", [1, 0])
def test_paper_snapshot_thresholds(rd_weight):
    # The snapshot runs of Sec. 6.4 / App. D use thresholds of a few 1e-3 (snap1004_1003: band
    # [1/1.004, 1.004], clip 0.003).  At that scale the decisions must still be
    # bit-exact away from the 1e-6 exemption, with a fifth of the tokens out of
    # band and a tenth clipped.
    b = make_loss_batch("tight_f32_v151936", T=512, seed=5, device="cuda")
    st, o = _full_parity(b, rd_weight=rd_weight, n_dz_rows=32)
    assert 0.05 * o["n_valid"] < o["n_rd_out"] < 0.5 * o["n_valid"]
    assert 0.03 * o["n_valid"] < o["n_clipped"] < 0.5 * o["n_valid"]
    assert np.count_nonzero(o["g"]) > 0.3 * o["n_valid"]   # the dlogits check is not vacuous
