"""K3 parity: occ_ewma_update against the float64 oracle (R10).

Tolerance: the parity bar's 1e-6 relative, taken relative to the magnitude of the
two terms of the App. B update, |a theta_prox| + |b theta| (which equals the
result's magnitude unless the terms cancel).  Resets and first steps from an
empty history must reproduce theta bit for bit.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import EWMA_N_7B, make_ewma_buffers

pytestmark = pytest.mark.gpu

RTOL = 1e-6


def _stats_tensor(n_active, n_valid):
    """A device occ_loss_stats with the given counters (other fields zero)."""
    import struct
    raw = struct.pack("<2d5q2i", 0.0, 0.0, n_valid, 0, 0, n_active, n_valid, 0, 0)
    return torch.frombuffer(bytearray(raw), dtype=torch.uint8).to("cuda")


def _check_step(tp_before, th, tp_after, a, b):
    ref = a * tp_before + b * th
    scale = np.abs(a * tp_before) + np.abs(b * th)
    err = np.abs(tp_after.astype(np.float64) - ref)
    assert np.all(err <= RTOL * scale + 1e-30), f"max rel {np.max(err / (scale + 1e-300)):.3g}"


@pytest.mark.parametrize("n", [1, 3, 4, 1000, 1_000_003])
@pytest.mark.parametrize("misalign", [0, 1])
def test_recursion_from_empty_history(n, misalign):
    beta = 0.75
    buf_th, buf_tp = make_ewma_buffers(n + misalign, seed=n, device="cuda")
    th, tp = buf_th[misalign:], buf_tp[misalign:]
    st = occ.new_ewma_state("cuda", w0=0.0)
    ost = oracle.EwmaState()
    ref = tp.cpu().numpy().astype(np.float64)
    g = torch.Generator(device="cuda").manual_seed(1)
    for step in range(5):
        before = tp.cpu().numpy().astype(np.float64)
        occ.occ_ewma_update(tp, th, beta, st)
        torch.cuda.synchronize()
        ref, ost, (a, b, reset) = oracle.ewma_update(ref, th.cpu().numpy(), beta, ost)
        got = tp.cpu().numpy()
        dst = occ.decode_ewma_state(st)
        assert abs(dst.w - ost.w) <= 1e-15 * ost.w and dst.streak == ost.streak
        if step == 0:  # w^(0) = 1: theta_prox^(0) = theta^(0) exactly (App. B)
            assert np.array_equal(got, th.cpu().numpy())
        else:
            _check_step(before, th.cpu().numpy().astype(np.float64), got, a, b)
        # next actor parameters
        th.add_(torch.randn(n, generator=g, device="cuda") * 1e-3)


def test_stationary_regime_matches_table1_plain_ewma():
    beta = 0.99
    th, tp = make_ewma_buffers(4_000_037, seed=3, device="cuda")
    st = occ.new_ewma_state("cuda", w0=1.0 / (1.0 - beta))
    before = tp.cpu().numpy().astype(np.float64)
    occ.occ_ewma_update(tp, th, beta, st)
    torch.cuda.synchronize()
    dst = occ.decode_ewma_state(st)
    assert abs(dst.coef_b - 0.01) < 1e-15 and abs(dst.coef_a - 0.99) < 1e-15
    _check_step(before, th.cpu().numpy().astype(np.float64), tp.cpu().numpy(), 0.99, 0.01)


def test_auto_reset_rule_on_device():
    beta, tau = 0.75, 0.9
    th, tp = make_ewma_buffers(100_000, seed=4, device="cuda")
    st = occ.new_ewma_state("cuda", w0=4.0)
    ost = oracle.EwmaState(w=4.0)
    seq = [(95, 100), (50, 100), (99, 100), (50, 100), (40, 100), (7, 0), (10, 100)]
    for n_act, n_val in seq:
        before = tp.cpu().numpy().astype(np.float64)
        occ.occ_ewma_update(tp, th, beta, st, stats=_stats_tensor(n_act, n_val), tau=tau,
                            min_streak=2)
        torch.cuda.synchronize()
        a, b, reset, ost = oracle.ewma_coefficients(ost, beta, n_active=n_act, n_valid=n_val,
                                                    tau=tau, min_streak=2)
        dst = occ.decode_ewma_state(st)
        assert (dst.streak, dst.n_resets, bool(dst.last_reset)) == (ost.streak, ost.n_resets, reset)
        if reset:
            assert np.array_equal(tp.cpu().numpy(), th.cpu().numpy())
        else:
            _check_step(before, th.cpu().numpy().astype(np.float64), tp.cpu().numpy(), a, b)
        th.add_(1e-3)
    assert ost.n_resets == 1
    occ.occ_ewma_update(tp, th, beta, st, force_reset=True)
    torch.cuda.synchronize()
    assert torch.equal(tp, th) and occ.decode_ewma_state(st).n_resets == 2


def test_constant_parameters_fixed_point_bitwise():
    th, _ = make_ewma_buffers(1 << 20, seed=5, device="cuda")
    tp = th.clone()
    st = occ.new_ewma_state("cuda", w0=7.0)
    for _ in range(3):
        occ.occ_ewma_update(tp, th, 0.9, st)
    torch.cuda.synchronize()
    assert torch.equal(tp, th)


def test_invalid_arguments():
    x = torch.zeros(8, device="cuda")
    st = occ.new_ewma_state("cuda")
    with pytest.raises(occ.OccError, match="invalid argument"):
        occ.occ_ewma_update(x, x, 0.5, st)          # theta_prox aliases theta
    with pytest.raises(occ.OccError, match="invalid argument"):
        occ.occ_ewma_update(x, x.clone(), 1.0, st)  # beta outside [0, 1)


@pytest.mark.slow
def test_full_size_7p6e9_sampled():
    """7.6e9-parameter buffers (61 GB on the device): sampled elements, the
    first and last million and the ragged tail against the oracle."""
    n = EWMA_N_7B
    th, tp = make_ewma_buffers(n, seed=0, device="cuda")
    rng = np.random.default_rng(0)
    idx = np.unique(np.concatenate([rng.integers(0, n, 1_000_000), np.arange(1_000_000),
                                    np.arange(n - 1_000_000, n)]))
    it = torch.as_tensor(idx, device="cuda")
    before = tp[it].cpu().numpy().astype(np.float64)
    thv = th[it].cpu().numpy().astype(np.float64)
    st = occ.new_ewma_state("cuda", w0=1.0 / (1.0 - 0.99))
    occ.occ_ewma_update(tp, th, 0.99, st)
    torch.cuda.synchronize()
    _check_step(before, thv, tp[it].cpu().numpy(), 0.99, 0.01)


def test_checkpoint_and_resume_reproduce_the_run():
    # The EWMA state is caller-owned (the proximal buffer and the 40-byte state
    # with w, the coefficients, the streak and the reset count): saving both
    # to the host and restoring them resumes the App. B recursion and the
    # Sec. 5.2 streak exactly where it stopped.
    n = 1_000_003
    rng = np.random.default_rng(9)
    thetas = [torch.from_numpy(rng.normal(0, 0.02, n).astype(np.float32)).to("cuda")
              for _ in range(5)]
    # low ratios at steps 1-2 (a streak that spans the checkpoint after step 1)
    # and at steps 3-4: resets at steps 2 and 4
    ratios = [(90, 100), (40, 100), (45, 100), (30, 100), (20, 100)]
    stats = [occ.new_loss_stats("cuda") for _ in ratios]
    for s, (act, val) in zip(stats, ratios):
        # stats with the given n_active / n_valid (layout of occ_loss_stats)
        buf = np.zeros(64, dtype=np.uint8)
        buf[16:24] = np.frombuffer(np.int64(val).tobytes(), np.uint8)   # n_valid
        buf[40:48] = np.frombuffer(np.int64(act).tobytes(), np.uint8)   # n_active
        s.copy_(torch.from_numpy(buf))
    tp0 = thetas[0].clone()

    def run(tp, st, steps):
        for k in steps:
            occ.occ_ewma_update(tp, thetas[k], 0.75, st, stats=stats[k], tau=0.5, min_streak=2)

    tp, st = tp0.clone(), occ.new_ewma_state("cuda")
    run(tp, st, range(5))
    torch.cuda.synchronize()

    tp2, st2 = tp0.clone(), occ.new_ewma_state("cuda")
    run(tp2, st2, range(2))
    ckpt = (tp2.cpu().clone(), st2.cpu().clone())      # checkpoint after two steps
    run(tp2, st2, range(2, 4))                         # progress that is thrown away
    tp3, st3 = ckpt[0].to("cuda"), ckpt[1].to("cuda")  # resume from the checkpoint
    run(tp3, st3, range(2, 5))
    torch.cuda.synchronize()
    assert torch.equal(tp3, tp) and torch.equal(st3, st)
    s = occ.decode_ewma_state(st)
    assert s.n_resets == 2 and s.streak == 0
    saved = occ.decode_ewma_state(ckpt[1])
    assert saved.streak == 1 and saved.n_resets == 0   # the step-2 reset needs the saved streak
