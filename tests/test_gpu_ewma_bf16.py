"""bf16 and host-resident PPO-EWMA buffers (occ_ewma_update_bf16, occ_ewma_update_host).

A bf16 buffer is a quantised code: the kernel's bits must equal the oracle's,
which forms the update in the kernel's precision (float32 fused multiply-add)
and rounds by definition (nearest-even, or stochastically with the SplitMix64
stream).  The host-resident variant must reproduce the device-resident one
bit for bit, across chunk boundaries.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_ewma_buffers

pytestmark = pytest.mark.gpu


def _bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("theta_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("seed", [0, 12345])
@pytest.mark.parametrize("n,offset", [(1_000_003, 0), (4096, 3), (7, 0)])
def test_bf16_buffer_matches_oracle_bits(theta_dtype, seed, n, offset):
    th32, tp32 = make_ewma_buffers(n + offset, seed=n, device="cuda")
    th = th32.to(theta_dtype)[offset:]
    tp = tp32.to(torch.bfloat16)[offset:]
    beta = 0.75
    st = occ.new_ewma_state("cuda", w0=3.0)
    ost = oracle.EwmaState(w=3.0)
    for step in range(3):
        before = _bits(tp)
        s = seed + step if seed else 0
        occ.occ_ewma_update_bf16(tp, th, beta, st, sr_seed=s)
        torch.cuda.synchronize()
        a, b, reset, ost = oracle.ewma_coefficients(ost, beta)
        ref = oracle.ewma_update_bf16(before, th.float().cpu().numpy(), np.float32(b), reset,
                                      seed=s)
        got = _bits(tp)
        assert np.array_equal(got, ref), (step, int(np.sum(got != ref)))
        th.add_(torch.full_like(th, 1e-3))


@pytest.mark.parametrize("seed", [0, 12345])
def test_infinities_and_nans_survive_the_update(seed):
    # Non-finite parameters stay non-finite: inf stays inf, NaN stays NaN (all
    # payloads, including one whose low bits alone are set and one with every
    # mantissa bit set), and their finite neighbours in the same 8-parameter
    # vector round exactly as the oracle does.
    n = 4096
    th32, tp32 = make_ewma_buffers(n, seed=9, device="cuda")
    special = {3: 0x7F800000, 10: 0xFF800000, 17: 0x7FC00000, 24: 0x7FFFFFFF, 31: 0x7F800001,
               40: 0xFFFFFFFF, 1000: 0x7F800000, 4095: 0x7FC00001}
    raw = th32.view(torch.int32)
    for i, b in special.items():
        raw[i] = b - (1 << 32) if b >= 1 << 31 else b
    tp = tp32.to(torch.bfloat16)
    before = _bits(tp)
    st = occ.new_ewma_state("cuda", w0=3.0)
    occ.occ_ewma_update_bf16(tp, th32, 0.75, st, sr_seed=seed)
    torch.cuda.synchronize()
    a, b, reset, _ = oracle.ewma_coefficients(oracle.EwmaState(w=3.0), 0.75)
    ref = oracle.ewma_update_bf16(before, th32.cpu().numpy(), np.float32(b), reset, seed=seed)
    got = _bits(tp)
    idx = np.array(sorted(special))
    finite = np.ones(n, dtype=bool)
    finite[idx] = False
    assert np.array_equal(got[finite], ref[finite])
    x = th32.cpu().numpy()[idx]
    assert np.all((got[idx] & 0x7F80) == 0x7F80)                     # still non-finite
    assert np.all(((got[idx] & 0x7F) != 0) == np.isnan(x))          # NaN iff NaN
    inf = np.isinf(x)
    assert np.array_equal(got[idx][inf], ref[idx][inf])              # infinities exact


def test_bf16_reset_copies_bf16_theta_exactly():
    th32, tp32 = make_ewma_buffers(100_000, seed=1, device="cuda")
    th = th32.to(torch.bfloat16)
    tp = tp32.to(torch.bfloat16)
    st = occ.new_ewma_state("cuda", w0=5.0)
    occ.occ_ewma_update_bf16(tp, th, 0.9, st, force_reset=True, sr_seed=7)
    torch.cuda.synchronize()
    assert torch.equal(tp, th)


def test_stochastic_rounding_keeps_small_steps():
    # beta = 0.99 in the stationary regime: b = 0.01, steps far below a bf16 ulp.
    n = 1 << 20
    tp = torch.full((n,), 1.0, dtype=torch.bfloat16, device="cuda")
    th = torch.full((n,), 1.0 + 2.0 ** -8, dtype=torch.float32, device="cuda")  # half a bf16 ulp up
    tp_rn = tp.clone()
    st = occ.new_ewma_state("cuda", w0=100.0)
    st2 = occ.new_ewma_state("cuda", w0=100.0)
    occ.occ_ewma_update_bf16(tp, th, 0.99, st, sr_seed=2024)
    occ.occ_ewma_update_bf16(tp_rn, th, 0.99, st2, sr_seed=0)
    torch.cuda.synchronize()
    exact = 1.0 + 0.01 * 2.0 ** -8
    assert torch.all(tp_rn == 1.0)                      # nearest rounding loses the step
    assert abs(tp.double().mean().item() - exact) < 2e-6  # stochastic rounding keeps it


@pytest.mark.parametrize("prox_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("staging_kb", [64, 4096])
def test_host_buffer_equals_device_buffer(prox_dtype, staging_kb):
    n = 3_000_017
    th, tp = make_ewma_buffers(n, seed=3, device="cuda")
    tp = tp.to(prox_dtype)
    dev = tp.clone()
    host = tp.cpu().pin_memory()
    st_d = occ.new_ewma_state("cuda", w0=2.0)
    st_h = occ.new_ewma_state("cuda", w0=2.0)
    staging = torch.empty(staging_kb * 1024, dtype=torch.uint8, device="cuda")
    s1 = torch.cuda.Stream()
    for step in range(3):
        seed = 11 + step if prox_dtype == torch.bfloat16 else 0
        if prox_dtype == torch.float32:
            occ.occ_ewma_update(dev, th, 0.8, st_d)
        else:
            occ.occ_ewma_update_bf16(dev, th, 0.8, st_d, sr_seed=seed)
        occ.occ_ewma_update_host(host, th, 0.8, st_h, staging, sr_seed=seed, stream1=s1)
        torch.cuda.synchronize()
        assert torch.equal(host, dev.cpu()), step
        th.mul_(0.999)
    assert torch.equal(st_d, st_h)


def test_host_buffer_rejects_pageable_memory():
    th = torch.zeros(16, device="cuda")
    st = occ.new_ewma_state("cuda")
    staging = torch.empty(1024, dtype=torch.uint8, device="cuda")
    lib = occ.lib()
    import ctypes
    pageable = torch.zeros(16)
    rc = lib.occ_ewma_update_host(ctypes.c_void_p(pageable.data_ptr()), 0,
                                  ctypes.c_void_p(th.data_ptr()), 0, 16, 0.5,
                                  ctypes.c_void_p(st.data_ptr()), None, 0.9, 1, 0, 0,
                                  ctypes.c_void_p(staging.data_ptr()), 1024, None, None)
    assert rc == 1 and b"pinned" in lib.occ_last_error()
