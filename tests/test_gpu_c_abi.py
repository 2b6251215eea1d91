"""The C ABI from a plain C program (tests/c_abi_caller.c): no PyTorch.

include/occ.h must compile as C11, and a C caller that allocates with
cudaMalloc and passes raw pointers must get the oracle's results: log pi_old
(R1), the loss, flags and dlogits (R2-R9), and one PPO-EWMA step whose
auto-reset reads the loss statistics on the device (R10).
"""

import os
import shutil
import subprocess

import numpy as np
import pytest

import oracle as orc
from paper_2605_12070_gb300 import build
from paper_2605_12070_gb300.workloads import make_loss_batch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _compile(out_dir):
    if shutil.which("gcc") is None or not os.path.exists(os.path.join(CUDA, "include",
                                                                      "cuda_runtime.h")):
        pytest.skip("gcc or the CUDA headers are missing")
    lib = build.build()
    exe = os.path.join(out_dir, "c_abi_caller")
    cmd = ["gcc", "-std=c11", "-O2", "-Wall", "-Wextra", "-Werror",
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
           os.path.join(ROOT, "tests", "c_abi_caller.c"), "-o", exe,
           "-L", os.path.dirname(lib), "-locc", "-L", os.path.join(CUDA, "lib64"), "-lcudart",
           "-Wl,-rpath," + os.path.dirname(lib)]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


def test_header_compiles_as_c11_and_links(tmp_path):
    _compile(str(tmp_path))


@pytest.mark.gpu
def test_c_caller_matches_the_oracle(tmp_path):
    d = str(tmp_path)
    exe = _compile(d)
    T, V, n = 64, 1000, 100_003
    b = make_loss_batch("tiny_f32_v4096", T=T, V=V, seed=3, device="cpu")
    z = b.z_theta.numpy().astype(np.float32)
    zo = b.z_old.numpy().astype(np.float32)
    ids = b.ids.numpy().astype(np.int32)
    lmu = b.logp_mu.numpy().astype(np.float32)
    rng = np.random.default_rng(3)
    adv = rng.standard_normal(T).astype(np.float32)
    mask = (rng.random(T) < 0.85).astype(np.uint8)
    th = rng.normal(0, 0.02, n).astype(np.float32)
    tp = (th + rng.normal(0, 1e-3, n)).astype(np.float32)
    for name, arr in (("z.f32", z), ("z_old.f32", zo), ("ids.i32", ids), ("lmu.f32", lmu),
                      ("adv.f32", adv), ("mask.u8", mask), ("theta.f32", th),
                      ("theta_prox.f32", tp)):
        arr.tofile(os.path.join(d, name))
    r = subprocess.run([exe, d, str(T), str(V), str(n)], capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stdout + r.stderr

    def read(name, dt, count):
        return np.fromfile(os.path.join(d, name), dtype=dt, count=count)

    # R1: log pi_old
    lo64, _ = orc.token_logprob(zo.astype(np.float64), ids.astype(np.int64))
    lt64, lse = orc.token_logprob(z.astype(np.float64), ids.astype(np.int64))
    assert np.abs(read("logp_old.f32", np.float32, T) - lo64).max() <= 1e-5
    # R2-R9 with log pi_old as the ABI passes it (float32)
    p = orc.LossParams(rd_lo=0.7, rd_hi=1.4, eps_low=0.2, eps_high=0.28, rd_weight=1)
    o = orc.token_terms(lt64, lo64.astype(np.float32).astype(np.float64), lmu, adv, mask, p)
    flags = read("flags.u8", np.uint8, T)
    near = np.minimum(o["dist_rd"], o["dist_rs"]) <= 1e-6
    assert not ((flags != o["flags"]) & ~near).any()
    stats = np.fromfile(os.path.join(d, "stats.bin"), dtype=np.uint8)
    loss = stats[8:16].view(np.float64)[0]
    n_valid, n_active = stats[16:24].view(np.int64)[0], stats[40:48].view(np.int64)[0]
    assert n_valid == o["n_valid"] and abs(loss - o["loss"]) <= 1e-4 * abs(o["loss"]) + 1e-12
    assert np.count_nonzero(o["g"]) > 0
    dz = read("dlogits.f32", np.float32, T * V).reshape(T, V)
    ok = ~((flags != o["flags"]) & near)
    ref = orc.softmax_grad_rows(z.astype(np.float64), ids.astype(np.int64), lse, o["g"])
    g = np.abs(o["g"])[:, None]
    assert np.all(np.abs(dz - ref)[ok] <= (2e-6 * np.abs(ref) + 4e-6 * g)[ok] + 1e-30)
    # R10: one step from the stationary state w = 1/(1 - beta); reset when rho < 0.5
    new, _, (a, bcoef, reset) = orc.ewma_update(tp.astype(np.float64), th.astype(np.float64),
                                                0.75, orc.EwmaState(w=4.0),
                                                n_active=int(n_active), n_valid=int(n_valid),
                                                tau=0.5)
    got = read("theta_prox_out.f32", np.float32, n).astype(np.float64)
    scale = np.abs(a * tp) + np.abs(bcoef * th)
    assert np.all(np.abs(got - new) <= 1e-6 * scale + 1e-30)
    assert ("loss" in r.stdout) and (n_active / n_valid < 0.5) == reset
