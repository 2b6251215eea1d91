"""K1 parity: occ_token_logprob against the float64 oracle (R1).

Tolerance: the parity bar's 2e-3 absolute on log-probabilities, plus a tight
bound derived from the kernel's arithmetic (float32 terms, compensated
merge, float64 epilogue, float32 output): |err| <= 1e-5.
"""

import numpy as np
import pytest
import torch

from kernel_choice import expected_kernel
from oracle_runner import logprob_rows
from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_loss_batch

pytestmark = pytest.mark.gpu

LOGP_TOL = 2e-3
LOGP_TIGHT = 1e-5


def _check(z, ids, rows=None, lse_too=True):
    logp, lse = occ.occ_token_logprob(z, ids, want_lse=lse_too)
    torch.cuda.synchronize()
    T = z.shape[0]
    rows = np.arange(T) if rows is None else np.asarray(rows)
    ref_lp, ref_lse = logprob_rows(z, ids, rows)
    got = logp.cpu().numpy().astype(np.float64)[rows]
    ok = np.isfinite(ref_lp)
    assert np.array_equal(np.isnan(got), ~ok)
    err = np.abs(got[ok] - ref_lp[ok])
    assert err.size == 0 or err.max() <= LOGP_TOL
    assert err.size == 0 or err.max() <= LOGP_TIGHT, f"max |dlogp| {err.max():.3g}"
    if lse_too:
        e2 = np.abs(lse.cpu().numpy().astype(np.float64)[rows] - ref_lse)
        assert e2.max() <= LOGP_TIGHT, f"max |dlse| {e2.max():.3g}"
    return err.max() if err.size else 0.0


@pytest.mark.parametrize("name,T", [("tiny_f32_v4096", 256), ("grpo_bf16_v32000", 300),
                                    ("agentic_bf16_v151936", 160),
                                    ("heavytail_bf16_v151936", 160)])
def test_workloads_reduced(name, T):
    b = make_loss_batch(name, T=T, seed=1, device="cuda")
    _check(b.z_old, b.ids)
    _check(b.z_theta, b.ids)


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [1, 2, 7, 8, 9, 31, 63, 65, 127, 129, 2040, 2048, 2056, 4095, 4097,
                               16376, 16384, 16392, 20000, 50000, 151936])
def test_vocab_edges(V, dtype):
    g = torch.Generator(device="cuda").manual_seed(V)
    T = 5
    z = (torch.randn((T, V), generator=g, device="cuda") * 3).to(dtype)
    ids = torch.tensor([0, V - 1, V // 2, 0, V - 1], dtype=torch.int32, device="cuda")
    _check(z, ids)
    assert occ.occ_last_kernel() == expected_kernel("k1", V, z.element_size())


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_strided_and_misaligned_rows(dtype):
    g = torch.Generator(device="cuda").manual_seed(7)
    big = (torch.randn((9, 5000), generator=g, device="cuda") * 2).to(dtype)
    ids = torch.randint(0, 4097, (9,), generator=g, device="cuda", dtype=torch.int32)
    vec_kernel = expected_kernel("k1", 4096, big.element_size())  # the aligned-row kernel
    _check(big[:, :4097], ids)        # ld = 5000 > V: aligned rows
    assert occ.occ_last_kernel() == vec_kernel
    _check(big[:, 1:4098], ids)       # base offset by one element: peeled rows
    assert occ.occ_last_kernel() == vec_kernel + "/peel"
    _check(big.reshape(-1)[: 9 * 4097].view(9, 4097), ids)  # ld = V = 4097: peeled rows
    assert occ.occ_last_kernel() == vec_kernel + "/peel"
    _check(big[:, 1:51], ids % 50)    # too short to peel: element loads
    assert occ.occ_last_kernel() == "k1_logprob_scalar"


@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("V", [4097, 20003])
def test_misaligned_rows_take_the_peeled_vector_kernel(dtype, V):
    g = torch.Generator(device="cuda").manual_seed(V)
    big = (torch.randn((17, V + 2), generator=g, device="cuda") * 2).to(dtype)
    z = big[:, 1:V + 1]                    # odd stride, every row-start residue
    ids = torch.randint(0, V, (17,), generator=g, device="cuda", dtype=torch.int32)
    ids[0], ids[-1] = 0, V - 1             # row 0's scalar prefix, the last row's tail
    _check(z, ids)
    assert occ.occ_last_kernel() == expected_kernel("k1", V, z.element_size())
    assert occ.occ_last_kernel().endswith("/peel")


def test_bad_ids_give_nan_and_empty():
    z = torch.randn((4, 100), device="cuda")
    ids = torch.tensor([-1, 100, 5, 99], dtype=torch.int32, device="cuda")
    logp, _ = occ.occ_token_logprob(z, ids)
    got = logp.cpu().numpy()
    assert np.isnan(got[:2]).all() and np.isfinite(got[2:]).all()
    e = torch.empty((0, 100), device="cuda")
    lp, _ = occ.occ_token_logprob(e, torch.empty(0, dtype=torch.int32, device="cuda"))
    assert lp.numel() == 0


def test_extreme_rows():
    # a one-hot row (+60), an all-equal row, a row with -inf entries
    V = 4096
    z = torch.zeros((3, V), device="cuda")
    z[0, 11] = 60.0
    z[2, : V // 2] = float("-inf")
    ids = torch.tensor([11, 3, V - 1], dtype=torch.int32, device="cuda")
    logp, lse = occ.occ_token_logprob(z, ids, want_lse=True)
    got = logp.cpu().numpy().astype(np.float64)
    assert abs(got[0] + np.log1p((V - 1) * np.exp(-60.0))) < 1e-6
    assert abs(got[1] + np.log(V)) < 1e-6
    assert abs(got[2] + np.log(V // 2)) < 1e-6


def test_full_size_agentic_sampled_rows():
    b = make_loss_batch("agentic_bf16_v151936", seed=0, device="cuda")
    rows = np.random.default_rng(0).choice(b.T, size=192, replace=False)
    rows = np.unique(np.concatenate([rows, [0, b.T - 1]]))
    _check(b.z_old, b.ids, rows=rows)
