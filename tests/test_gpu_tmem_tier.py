"""The tensor-memory tiers of the fused kernel and of K2 against their plain
kernels, bit for bit.

Long aligned rows keep 128 KB of the current row in tensor memory instead of
re-reading it from L2, and the kernel runs persistent with rows fetched from a
counter.  The arithmetic is the plain kernel's in the same order, so every
output must equal the plain kernel's (OCC_OPT_FUSED_TMEM / OCC_OPT_K2_TMEM = 0)
bit for bit: dlogits, the statistics, the log-probabilities and the flags.  The
oracle comparisons of the default paths (test_gpu_fused.py, test_gpu_loss.py,
test_gpu_full_agentic.py) run these tiers on the long-row batches.
"""

import pytest
import torch

from kernel_choice import expected_kernel
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu


def _both(b, **kw):
    outs = []
    for tm in (1, 0):
        with occ.options(fused_tmem=tm):
            out = occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv,
                                               b.mask, **b.thresholds(), **kw)
            kern = occ.occ_last_kernel()
        torch.cuda.synchronize()
        outs.append((out, kern))
    return outs


def _bits(t):
    return t.view(torch.int32) if t.dtype == torch.float32 else \
        t.view(torch.int16) if t.dtype == torch.bfloat16 else t


def _same(a, b):
    # bit patterns, so that the NaN of a dropped token's log-probability compares equal
    for k in ("stats", "logp", "logp_old", "flags", "dlogits"):
        if a.get(k) is not None or b.get(k) is not None:
            assert torch.equal(_bits(a[k]), _bits(b[k])), k


@pytest.mark.parametrize("T", [1, 3, 300, 1500])
def test_tmem_tier_equals_plain_kernel(T):
    # fewer rows than CTAs, a few rounds of the row counter, and many
    b = make_loss_batch("agentic_bf16_v151936", T=T, seed=T, device="cuda")
    (tm, ktm), (pl, kpl) = _both(b)
    assert ktm == "k2_fused_l2/tmem" and kpl == "k2_fused_l2"
    _same(tm, pl)


@pytest.mark.parametrize("variant", ["f32_logits", "f32_dlogits", "forward_only", "in_place",
                                     "bad_ids_and_masked"])
def test_tmem_tier_variants(variant):
    name = "tight_f32_v151936" if variant == "f32_logits" else "agentic_bf16_v151936"
    b = make_loss_batch(name, T=96, seed=11, device="cuda")
    kw = {}
    if variant == "f32_dlogits":
        kw = dict(dlogits_f32=True)
    elif variant == "forward_only":
        kw = dict(dlogits=None)
    elif variant == "bad_ids_and_masked":
        b.ids[3] = -1
        b.ids[40] = b.V
        b.mask[10:30] = 0
    if variant == "in_place":
        outs = []
        for tm in (1, 0):
            z = b.z_theta.clone()
            with occ.options(fused_tmem=tm):
                out = occ.occ_decoupled_loss_fused(z, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                                   dlogits="inplace", **b.thresholds())
                kern = occ.occ_last_kernel()
            torch.cuda.synchronize()
            outs.append((out, kern, z))
        assert outs[0][1] == "k2_fused_l2/tmem" and outs[1][1] == "k2_fused_l2"
        assert torch.equal(outs[0][2], outs[1][2])
        _same(outs[0][0], outs[1][0])
        return
    (tm, ktm), (pl, kpl) = _both(b, **kw)
    assert ktm == "k2_fused_l2/tmem" and kpl == "k2_fused_l2"
    _same(tm, pl)
    if variant == "bad_ids_and_masked":
        st = occ.decode_loss_stats(tm["stats"])
        m = b.mask.bool()
        m[3] = m[40] = False
        assert st.err == occ.DATA_ERR_BAD_ID and st.n_valid == int(m.sum())


@pytest.mark.parametrize("V", [98304, 114688, 114696])
def test_tmem_tier_threshold(V):
    # 98304 bf16 rows (192 KB) hold 24 blocks in whole rounds: the plain kernel;
    # 114688 hold 28 (the tier); 114696 one vector more (the walk's last round)
    b = make_loss_batch("agentic_bf16_v151936", T=40, V=V, seed=V, device="cuda")
    (tm, ktm), (pl, kpl) = _both(b)
    assert ktm == expected_kernel("fused", V, 2, diag=False) and kpl == "k2_fused_l2"
    assert ktm == ("k2_fused_l2" if V == 98304 else "k2_fused_l2/tmem")
    _same(tm, pl)


def test_diagnostics_tier_equals_plain_kernel():
    # the entropy / KL outputs: the same tier with 3 row pairs in flight
    b = make_loss_batch("agentic_bf16_v151936", T=200, seed=2, device="cuda")
    (tm, ktm), (pl, kpl) = _both(b, want_diagnostics=True)
    assert ktm == "k2_fused_l2/tmem" and kpl == "k2_fused_l2"
    _same(tm, pl)
    assert torch.equal(_bits(tm["entropy"]), _bits(pl["entropy"]))
    assert torch.equal(_bits(tm["kl"]), _bits(pl["kl"]))


def test_shape_options_keep_the_plain_kernels():
    b = make_loss_batch("agentic_bf16_v151936", T=16, seed=2, device="cuda")
    with occ.options(fused_head_bytes=65536):
        occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                     **b.thresholds())
        assert occ.occ_last_kernel() == "k2_fused_l2"
    with occ.options(fused_threads=512):
        occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                     **b.thresholds())
        assert occ.occ_last_kernel() == "k2_fused_l2"
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    for opt in (dict(k2_threads=512), dict(k2_head_bytes=65536), dict(k2_unroll=8)):
        with occ.options(**opt):
            occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                           **b.thresholds())
            assert occ.occ_last_kernel() == "k2_loss_l2", opt
    torch.cuda.synchronize()


def _k2_both(b, lp_old, **kw):
    outs = []
    for tm in (1, 0):
        with occ.options(k2_tmem=tm):
            out = occ.occ_decoupled_loss_fwd_bwd(b.z_theta, b.ids, lp_old, b.logp_mu, b.adv, b.mask,
                                                 **b.thresholds(), **kw)
            kern = occ.occ_last_kernel()
        torch.cuda.synchronize()
        outs.append((out, kern))
    return outs


@pytest.mark.parametrize("variant", ["plain", "few_rows", "many_rows", "f32_logits", "f32_dlogits",
                                     "forward_only", "bad_ids_and_masked", "proxy"])
def test_k2_tmem_tier_equals_plain_kernel(variant):
    name = "tight_f32_v151936" if variant == "f32_logits" else "agentic_bf16_v151936"
    T = {"few_rows": 3, "many_rows": 1500}.get(variant, 96)
    b = make_loss_batch(name, T=T, seed=13, device="cuda")
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    kw = {}
    if variant == "f32_dlogits":
        kw = dict(dlogits_f32=True)
    elif variant == "forward_only":
        kw = dict(dlogits=None)
    elif variant == "proxy":
        kw = dict(proxy="arithmetic", alpha=0.5)
    elif variant == "bad_ids_and_masked":
        b.ids[3] = -1
        b.mask[10:30] = 0
    (tm, ktm), (pl, kpl) = _k2_both(b, lp_old, **kw)
    assert ktm == "k2_loss_l2/tmem" and kpl == "k2_loss_l2"
    _same(tm, pl)


@pytest.mark.parametrize("V", [131064, 131072, 131080])
def test_k2_tmem_tier_threshold(V):
    # K2 walks 8 blocks per round: 131064 bf16 rows (16383 vectors) hold 24 blocks
    # in whole rounds (the plain kernel), 131072 hold 32 (the tier), 131080 one
    # vector more
    b = make_loss_batch("agentic_bf16_v151936", T=24, V=V, seed=V, device="cuda")
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    (tm, ktm), (pl, kpl) = _k2_both(b, lp_old)
    assert ktm == expected_kernel("k2", V, 2) and kpl == "k2_loss_l2"
    assert ktm == ("k2_loss_l2" if V == 131064 else "k2_loss_l2/tmem")
    _same(tm, pl)


@pytest.mark.parametrize("V,T", [(32000, 600), (32000, 2), (24000, 300), (16384, 100),
                                 (50000, 300), (40000, 5)])
def test_short_row_tier_equals_plain_kernels(V, T):
    # the 128-thread tier (64 columns per CTA, eight CTAs per SM) and the 256-thread
    # tier (128 columns, four per SM: V = 40000 and 50000 bf16)
    name = "tiny_f32_v4096" if V == 16384 else "grpo_bf16_v32000"
    b = make_loss_batch(name, T=T, V=V, seed=V + T, device="cuda")
    es = b.z_theta.element_size()
    (tm, ktm), (pl, kpl) = _both(b)
    assert ktm == expected_kernel("fused", V, es, diag=False) == "k2_fused_l2/tmem"
    assert kpl == "k2_fused_l2"
    _same(tm, pl)
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    (tm, ktm), (pl, kpl) = _k2_both(b, lp_old)
    assert ktm == expected_kernel("k2", V, es) and kpl == "k2_loss_l2"
    assert ktm == ("k2_loss_l2" if V == 24000 else "k2_loss_l2/tmem")
    _same(tm, pl)


@pytest.mark.parametrize("V", [151937, 50257, 32001])
def test_peeled_rows_tier_equals_plain_kernels(V):
    # rows with an odd stride start at every residue modulo 16 bytes: the peeled
    # kernels, in the 512-, 256- and 128-thread tiers
    b = make_loss_batch("agentic_bf16_v151936", T=40, V=V, seed=V, device="cuda")
    assert b.z_theta.stride(0) % 2 == 1
    (tm, ktm), (pl, kpl) = _both(b)
    assert ktm == expected_kernel("fused", V, 2, diag=False) == "k2_fused_l2/peel/tmem"
    assert kpl == "k2_fused_l2/peel"
    _same(tm, pl)
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    (tm, ktm), (pl, kpl) = _k2_both(b, lp_old)
    assert ktm == expected_kernel("k2", V, 2) == "k2_loss_l2/peel/tmem" and kpl == "k2_loss_l2/peel"
    _same(tm, pl)


def test_tmem_kernels_on_two_streams_at_once():
    # a fused and a K2 launch of the tier on two streams may share SMs: their CTAs'
    # tensor memory (NT / 2 columns each) fits the SM whenever their registers do
    b = make_loss_batch("agentic_bf16_v151936", T=1200, seed=21, device="cuda")
    g = make_loss_batch("grpo_bf16_v32000", T=3000, seed=22, device="cuda")
    lp_old, _ = occ.occ_token_logprob(g.z_old, g.ids)
    torch.cuda.synchronize()
    ref_f = occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                         **b.thresholds())
    ref_k = occ.occ_decoupled_loss_fwd_bwd(g.z_theta, g.ids, lp_old, g.logp_mu, g.adv, g.mask,
                                           **g.thresholds())
    torch.cuda.synchronize()
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    outs = []
    for _ in range(3):
        with torch.cuda.stream(s1):
            f = occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                             **b.thresholds())
        with torch.cuda.stream(s2):
            k = occ.occ_decoupled_loss_fwd_bwd(g.z_theta, g.ids, lp_old, g.logp_mu, g.adv, g.mask,
                                               **g.thresholds())
        outs.append((f, k))
    torch.cuda.synchronize()
    for f, k in outs:
        _same(f, ref_f)
        _same(k, ref_k)


def test_tmem_tiers_with_every_token_masked():
    # no row is read: the CTAs allocate, fetch rows, write zero gradients and free
    b = make_loss_batch("agentic_bf16_v151936", T=64, seed=31, device="cuda")
    b.mask.zero_()
    (tm, ktm), (pl, kpl) = _both(b)
    assert ktm == "k2_fused_l2/tmem"
    _same(tm, pl)
    assert torch.all(tm["dlogits"] == 0)
    st = occ.decode_loss_stats(tm["stats"])
    assert st.n_valid == 0 and st.loss == 0.0
    lp_old, _ = occ.occ_token_logprob(b.z_old, b.ids)
    (tm, ktm), (pl, kpl) = _k2_both(b, lp_old)
    assert ktm == "k2_loss_l2/tmem"
    _same(tm, pl)
    assert torch.all(tm["dlogits"] == 0)
