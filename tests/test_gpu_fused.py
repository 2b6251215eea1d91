"""occ_decoupled_loss_fused against the float64 oracle (R1..R9, R11).

In the fused kernel log pi_old never crosses the ABI, so the oracle chain
keeps it in float64 too.  Bars as in test_gpu_loss.py; the diagnostics
(entropy of pi_theta, KL(pi_old || pi_theta)) are checked to 1e-4 absolute
(float32 weighted sums of O(10) logits, float64 epilogue).
"""

import numpy as np
import pytest
import torch

import oracle as orc
from kernel_choice import expected_kernel
from oracle_runner import dlogits_rows, fp32, logprob_rows, loss_params, oracle_loss
from oracle.rows import to_f64
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import LossBatch, make_loss_batch

pytestmark = pytest.mark.gpu

EXEMPT = 1e-6
DIAG_TOL = 1e-4


def _oracle_diag(b, rows):
    it = torch.as_tensor(rows, device=b.z_theta.device)
    z = to_f64(b.z_theta[it])
    zo = to_f64(b.z_old[it])
    return orc.token_entropy(z), orc.token_kl(zo, z)


def _check_fused(b, out, rows_dz=None, f32=False, diag=True, require_grad=True):
    T = b.T
    rows = np.arange(T)
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    o = oracle_loss(b, lt64, lo64, loss_params(b))
    st = occ.decode_loss_stats(out["stats"])
    v = o["valid"]
    assert st.denom == o["N"] and st.n_valid == o["n_valid"] and st.err == 0
    fl = out["flags"].cpu().numpy()
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= EXEMPT
    diff = fl != o["flags"]
    assert not (diff & ~(near & v)).any()
    if not diff.any():
        assert (st.n_rd_out, st.n_clipped, st.n_active) == (o["n_rd_out"], o["n_clipped"],
                                                            o["n_active"])
    assert abs(st.loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
    if v.any():
        assert np.abs(out["logp"].cpu().numpy()[v] - lt64[v]).max() <= 1e-5
        assert np.abs(out["logp_old"].cpu().numpy()[v] - lo64[v]).max() <= 1e-5
    if diag:
        H, K = _oracle_diag(b, rows)
        gh = out["entropy"].cpu().numpy()
        gk = out["kl"].cpu().numpy()
        assert np.abs(gh[v] - H[v]).max() <= DIAG_TOL
        assert np.abs(gk[v] - K[v]).max() <= DIAG_TOL
        assert np.all(gh[~v] == 0) and np.all(gk[~v] == 0)
    if rows_dz is None:
        act = np.nonzero(o["g"] != 0)[0]
        rows_dz = np.unique(np.concatenate([act[:24], [0, T - 1]]))
    rows_dz = np.array([r for r in rows_dz if not diff[r]], dtype=np.int64)
    if require_grad and o["n_valid"] > 0:  # the batch must exercise the gradient
        assert np.count_nonzero(o["g"][rows_dz]) > 0, "no compared row carries a gradient"
    ref = dlogits_rows(b, rows_dz, lse[rows_dz], o["g"][rows_dz])
    got = out["dlogits"][torch.as_tensor(rows_dz, device="cuda")].float().cpu().numpy()
    g = np.abs(o["g"][rows_dz])[:, None]
    rel = 2e-6 if (f32 or b.z_theta.dtype == torch.float32) else 2.0 ** -8
    err = np.abs(got - ref)
    assert err.max() <= 3e-3
    assert np.all(err <= rel * np.abs(ref) + 4e-6 * g + 1e-30)
    return st, o


def _fused(b, **kw):
    out = occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                       **b.thresholds(), **kw)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("name,T", [("tiny_f32_v4096", 256), ("grpo_bf16_v32000", 600),
                                    ("agentic_bf16_v151936", 300),
                                    ("heavytail_bf16_v151936", 300),
                                    ("tight_f32_v151936", 384)])
@pytest.mark.parametrize("diag", [True, False])
def test_fused_workloads(name, T, diag):
    b = make_loss_batch(name, T=T, seed=4, device="cuda")
    out = _fused(b, want_diagnostics=diag)
    _check_fused(b, out, diag=diag)


def test_fused_f32_dlogits_and_grad_scale():
    b = make_loss_batch("agentic_bf16_v151936", T=256, seed=5, device="cuda")
    out = _fused(b, dlogits_f32=True, grad_scale=1000.0, want_diagnostics=True)
    lo64, _ = logprob_rows(b.z_old, b.ids, np.arange(b.T))
    lt64, lse = logprob_rows(b.z_theta, b.ids, np.arange(b.T))
    o = oracle_loss(b, lt64, lo64, loss_params(b, grad_scale=1000.0))
    act = np.nonzero(o["g"] != 0)[0][:16]
    ref = dlogits_rows(b, act, lse[act], o["g"][act])
    got = out["dlogits"][torch.as_tensor(act, device="cuda")].cpu().numpy()
    assert np.all(np.abs(got - ref) <= 2e-6 * np.abs(ref) + 4e-6 * np.abs(o["g"][act])[:, None])


def test_fused_matches_two_call_sequence():
    b = make_loss_batch("agentic_bf16_v151936", T=512, seed=6, device="cuda")
    fused = _fused(b)
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    seq = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                         **b.thresholds())
    torch.cuda.synchronize()
    v = (fused["flags"] & occ.FLAG_VALID) != 0
    assert (fused["logp"][v] - seq["logp"][v]).abs().max().item() <= 2e-6
    assert (fused["logp_old"][v] - lp_old[v]).abs().max().item() <= 2e-6
    same = fused["flags"] == seq["flags"]
    assert same.float().mean().item() > 0.999
    d = (fused["dlogits"][same].float() - seq["dlogits"][same].float()).abs()
    assert d.max().item() <= 2.0 ** -7 * seq["dlogits"][same].float().abs().max().item()


@pytest.mark.parametrize("layout", ["offset", "ld_odd", "old_padded"])
def test_fused_strided_and_misaligned(layout):
    g = torch.Generator(device="cuda").manual_seed(3)
    T, V = 19, 3001
    extra = {"offset": 9, "ld_odd": 2, "old_padded": 0}[layout]
    bufz = (torch.randn((T, V + extra + 1), generator=g, device="cuda") * 2).to(torch.bfloat16)
    z = bufz[:, 1:V + 1] if layout == "offset" else bufz[:, :V]
    old_ld = V + (7 if layout == "old_padded" else extra + 1)
    bufo = torch.empty((T, old_ld), dtype=torch.bfloat16, device="cuda")
    bufo[:, :V] = (z.float() + 0.3 * torch.randn((T, V), generator=g, device="cuda")).to(
        torch.bfloat16)
    zo = bufo[:, :V]
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    lo64, _ = logprob_rows(zo, ids, np.arange(T))
    lmu = torch.from_numpy(fp32(lo64 + np.random.default_rng(3).normal(0, 0.2, T))).cuda()
    b = LossBatch("edge", z, zo, ids, lmu, torch.randn(T, generator=g, device="cuda"),
                  (torch.rand(T, generator=g, device="cuda") < 0.8).to(torch.uint8),
                  rd_lo=0.7, rd_hi=1.4)
    out = _fused(b, want_diagnostics=True)
    assert occ.occ_last_kernel() == "k2_fused_stream"  # rows at different byte offsets
    _check_fused(b, out, rows_dz=np.arange(T))


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("diag", [True, False])
def test_fused_misaligned_rows_with_matching_layouts(dtype, diag):
    """Current, old and gradient rows all one element past a 16-byte boundary
    with one odd stride: the peeled vector kernel, every row-start residue,
    the sampled token in row 0's scalar prefix and in the last row's tail."""
    g = torch.Generator(device="cuda").manual_seed(13)
    T, V, off = 23, 3001, 1
    ld = V + 2
    bz, bo = (torch.empty((T, ld), dtype=dtype, device="cuda") for _ in range(2))
    bd = torch.full((T, ld), 7.0, dtype=dtype, device="cuda")
    z, zo, dz = bz[:, off:off + V], bo[:, off:off + V], bd[:, off:off + V]
    z.copy_((torch.randn((T, V), generator=g, device="cuda") * 2).to(dtype))
    zo.copy_((z.float() + 0.3 * torch.randn((T, V), generator=g, device="cuda")).to(dtype))
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    ids[0], ids[-1] = 0, V - 1
    lo64, _ = logprob_rows(zo, ids, np.arange(T))
    lmu = torch.from_numpy(fp32(lo64 + np.random.default_rng(13).normal(0, 0.2, T))).cuda()
    b = LossBatch("edge", z, zo, ids, lmu, torch.randn(T, generator=g, device="cuda"),
                  (torch.rand(T, generator=g, device="cuda") < 0.8).to(torch.uint8),
                  rd_lo=0.7, rd_hi=1.4)
    b.mask[0] = b.mask[-1] = 1
    out = _fused(b, dlogits=dz, want_diagnostics=diag)
    assert occ.occ_last_kernel() == "k2_fused_l2/peel"
    out["dlogits"] = dz
    _check_fused(b, out, rows_dz=np.arange(T), diag=diag)
    assert torch.all(bd[:, :off] == 7.0) and torch.all(bd[:, off + V:] == 7.0)


def test_fused_in_place_bad_ids_and_empty():
    b = make_loss_batch("grpo_bf16_v32000", T=64, seed=8, device="cuda")
    ref = _fused(b)
    z2 = b.z_theta.clone()
    out = occ.occ_decoupled_loss_fused(z2, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                       dlogits="inplace", **b.thresholds())
    torch.cuda.synchronize()
    assert torch.equal(z2, ref["dlogits"]) and torch.equal(out["stats"], ref["stats"])
    b.ids[5] = -3
    out = _fused(b, want_diagnostics=True)
    st = occ.decode_loss_stats(out["stats"])
    assert st.err == occ.DATA_ERR_BAD_ID and st.n_valid == 63
    assert torch.isnan(out["logp_old"][5]) and torch.all(out["dlogits"][5] == 0)
    e = torch.empty((0, 100), device="cuda")
    i0 = torch.empty(0, dtype=torch.int32, device="cuda")
    f0 = torch.empty(0, device="cuda")
    out = occ.occ_decoupled_loss_fused(e, e, i0, f0, f0, None, rd_lo=0.5, rd_hi=2.0,
                                       eps_low=0.2, eps_high=0.28)
    assert occ.decode_loss_stats(out["stats"]).denom == 0


def test_fused_full_size_agentic_sampled():
    """The bench workload through the fused kernel, sampled rows against the oracle."""
    b = make_loss_batch("agentic_bf16_v151936", seed=0, device="cuda")
    out = _fused(b, want_diagnostics=True)
    mask = b.mask.cpu().numpy()
    rng = np.random.default_rng(2)
    rows = np.unique(np.concatenate([rng.choice(np.nonzero(mask)[0], 128, replace=False),
                                     [0, b.T - 1]]))
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    o = orc.token_terms(lt64, lo64, b.logp_mu.cpu().numpy()[rows], b.adv.cpu().numpy()[rows],
                        mask[rows], loss_params(b), N=int(mask.sum()))
    fl = out["flags"].cpu().numpy()[rows]
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= EXEMPT
    assert not ((fl != o["flags"]) & ~near).any()
    v = o["valid"]
    assert np.abs(out["logp_old"].cpu().numpy()[rows][v] - lo64[v]).max() <= 1e-5
    H, K = _oracle_diag(b, rows)
    assert np.abs(out["entropy"].cpu().numpy()[rows][v] - H[v]).max() <= DIAG_TOL
    assert np.abs(out["kl"].cpu().numpy()[rows][v] - K[v]).max() <= DIAG_TOL


def test_fused_odd_vocab_past_2_31_logits_sampled():
    """An odd vocabulary (ld = V = 50257: rows off 16-byte boundaries, the
    peeled kernel and its tensor-memory tier) over more than 2^31 logits per
    tensor, so row offsets pass 4 GB; sampled rows (the first, the last, random
    ones) against the oracle, dlogits included."""
    b = make_loss_batch("grpo_bf16_v32000", T=45_000, V=50_257, seed=6, device="cuda")
    T, V = b.T, b.V
    assert T * V > 2 ** 31
    out = _fused(b)
    # the peeled rows of the 256-thread tier keep 64 KB each in tensor memory
    assert occ.occ_last_kernel() == expected_kernel("fused", V, 2, diag=False) == \
        "k2_fused_l2/peel/tmem"
    mask = np.ones(T, np.uint8) if b.mask is None else b.mask.cpu().numpy()
    rng = np.random.default_rng(6)
    rows = np.unique(np.concatenate([rng.choice(T, 96, replace=False), [0, 1, T - 2, T - 1]]))
    lo64, _ = logprob_rows(b.z_old, b.ids, rows)
    lt64, lse = logprob_rows(b.z_theta, b.ids, rows)
    o = orc.token_terms(lt64, lo64, b.logp_mu.cpu().numpy()[rows], b.adv.cpu().numpy()[rows],
                        mask[rows], loss_params(b), N=int(mask.sum()))
    fl = out["flags"].cpu().numpy()[rows]
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= EXEMPT
    assert not ((fl != o["flags"]) & ~near).any()
    v = o["valid"]
    assert np.abs(out["logp"].cpu().numpy()[rows][v] - lt64[v]).max() <= 1e-5
    assert np.abs(out["logp_old"].cpu().numpy()[rows][v] - lo64[v]).max() <= 1e-5
    keep = fl == o["flags"]
    assert np.count_nonzero(o["g"][keep]) > 0
    ref = dlogits_rows(b, rows[keep], lse[keep], o["g"][keep])
    got = out["dlogits"][torch.as_tensor(rows[keep], device="cuda")].float().cpu().numpy()
    g = np.abs(o["g"][keep])[:, None]
    assert np.all(np.abs(got - ref) <= 2.0 ** -8 * np.abs(ref) + 4e-6 * g + 1e-30)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [1, 7, 8, 9, 63, 65, 127, 129, 4095, 4097, 8184, 8192, 8200, 16376,
                               16384, 16392, 20000, 50000, 65536, 65536 + 3, 65544])
def test_fused_vocab_edges(V, dtype):
    # rows shorter than one vector, one vector exactly, a ragged tail after the
    # vector body, rows in each CTA-size tier (40 / 80 / 100 / 200 KB) and rows
    # longer than the shared-memory head (65539 bf16 = 128 KB)
    g = torch.Generator(device="cuda").manual_seed(V)
    T = 37
    z = (torch.randn((T, V), generator=g, device="cuda") * 2.5).to(dtype)
    zo = (z.float() + 0.3 * torch.randn((T, V), generator=g, device="cuda")).to(dtype)
    ids = torch.randint(0, V, (T,), generator=g, device="cuda", dtype=torch.int32)
    ids[0], ids[-1] = 0, V - 1
    lo64, _ = logprob_rows(zo, ids, np.arange(T))
    lmu = torch.from_numpy(fp32(lo64 + np.random.default_rng(V).normal(0, 0.3, T))).cuda()
    b = LossBatch("edge", z, zo, ids, lmu, torch.randn(T, generator=g, device="cuda"),
                  (torch.rand(T, generator=g, device="cuda") < 0.8).to(torch.uint8),
                  rd_lo=0.7, rd_hi=1.4)
    out = _fused(b, want_diagnostics=True)
    assert occ.occ_last_kernel() == expected_kernel("fused", V, z.element_size())
    _check_fused(b, out, rows_dz=np.arange(T))
    if V == 1:  # a one-token vocabulary: log pi = 0, entropy 0, KL 0
        v = b.mask.cpu().numpy().astype(bool)
        assert np.all(np.abs(out["logp"].cpu().numpy()[v]) <= 1e-5)
        assert np.all(np.abs(out["entropy"].cpu().numpy()[v]) <= 1e-6)
        assert np.all(np.abs(out["kl"].cpu().numpy()[v]) <= 1e-6)
