"""Host-side checks of the C-ABI library that need no GPU.

The library must load, export every entry point include/occ.h declares, and
reject invalid calls on the host before touching the device.
"""

import ctypes
import os
import re

import pytest

from paper_2605_12070_gb300 import build, occ

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return occ.lib()


def _declared_symbols():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(occ_[a-z0-9_]+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported(L):
    declared = _declared_symbols()
    assert {"occ_token_logprob", "occ_decoupled_loss_fwd_bwd", "occ_ewma_update"} <= declared
    for name in declared:
        assert hasattr(L, name), name
    assert declared <= set(occ.EXPORTS)


def test_version_and_status_strings(L):
    assert L.occ_version() == 1
    assert L.occ_status_string(0) == b"ok"
    assert L.occ_status_string(5).startswith(b"workspace")


def test_host_validation_without_gpu(L):
    null = ctypes.c_void_p(0)
    # V = 0 is rejected before any CUDA call
    rc = L.occ_token_logprob(null, 0, 4, 0, 0, null, null, null, null)
    assert rc == 1 and b"V >= 1" in L.occ_last_error()
    # T = 0 is a no-op and launches nothing
    assert L.occ_token_logprob(null, 1, 0, 10, 10, null, null, null, null) == 0
    assert L.occ_last_kernel() == b""
    # bad dtype
    assert L.occ_token_logprob(null, 7, 1, 10, 10, null, null, null, null) == 2
    # a vocabulary that int32 ids cannot index
    big = 2 ** 31
    assert L.occ_token_logprob(null, 1, 1, big, big, null, null, null, null) == 2
    assert b"exceeds" in L.occ_last_error()
    # inverted band
    p = occ.LossParams(2.0, 1.0, 0.2, 0.28, 1.0, 0, 1, 0)
    rc = L.occ_decoupled_loss_fwd_bwd(null, 1, 1, 8, 8, null, null, null, null, null,
                                      ctypes.byref(p), null, null, null, 0, null, null, 0, null)
    assert rc == 1
    # missing workspace
    p = occ.LossParams(0.5, 2.0, 0.2, 0.28, 1.0, 0, 1, 0)
    stats = ctypes.create_string_buffer(64)
    rc = L.occ_decoupled_loss_fwd_bwd(null, 1, 1, 8, 8, null, null, null, null, null,
                                      ctypes.byref(p), null, null, null, 0,
                                      ctypes.cast(stats, ctypes.c_void_p), null, 0, null)
    assert rc == 5
    # allocation-free loss: a null params pointer and a negative T are argument
    # errors before the size limit is looked at; only then is a T beyond the
    # scratch array unsupported (all before any CUDA call)
    nf = L.occ_decoupled_loss_fwd_bwd_noalloc
    big_T = occ.NOALLOC_MAX_TOKENS + 1
    assert nf(null, 1, big_T, 8, 8, null, null, null, null, null, None, null, null, null, 0,
              null, null) == 1
    assert b"params" in L.occ_last_error()
    assert nf(null, 1, -1, 8, 8, null, null, null, null, null, ctypes.byref(p), null, null, null,
              0, null, null) == 1
    assert nf(null, 1, big_T, 8, 8, null, null, null, null, null, ctypes.byref(p), null, null,
              null, 0, null, null) == 2
    assert b"at most" in L.occ_last_error()
    # EWMA: beta out of range, min_streak < 1
    st = ctypes.create_string_buffer(48)
    stp = ctypes.cast(st, ctypes.c_void_p)
    assert L.occ_ewma_update(null, null, 0, 1.5, stp, null, 0.9, 1, 0, null) == 1
    assert L.occ_ewma_update(null, null, 0, 0.5, stp, null, 0.9, 0, 0, null) == 1


def test_workspace_size_grows_with_tokens(L):
    a = occ.occ_loss_workspace_bytes(0, 151936)
    b = occ.occ_loss_workspace_bytes(65536, 151936)
    assert 0 < a < b and b >= 65536 * 5 and b % 256 == 0


def test_no_cpu_fallback():
    import torch
    with pytest.raises(occ.OccError, match="CUDA"):
        occ.occ_token_logprob(torch.zeros(2, 4), torch.zeros(2, dtype=torch.int32))


def test_host_alloc_argument_checks(L):
    p = ctypes.c_void_p(1)
    assert L.occ_host_alloc(0, ctypes.byref(p)) == 1 and p.value is None
    assert b"bytes == 0" in L.occ_last_error()
    assert L.occ_host_alloc(1 << 20, None) == 1
    assert L.occ_host_free(None, 0) == 0
    assert L.occ_host_free(ctypes.c_void_p(4096 + 1), 1 << 20) == 1  # not from occ_host_alloc


def test_host_alloc_fails_cleanly_without_a_device(L):
    import torch
    if torch.cuda.is_available():
        pytest.skip("a device is present")
    p = ctypes.c_void_p()
    assert L.occ_host_alloc(1 << 20, ctypes.byref(p)) == 4  # OCC_ERR_CUDA
    assert p.value is None and b"cudaHostRegister" in L.occ_last_error()


def test_error_messages_are_per_host_thread(L):
    # occ_last_error is documented per host thread: a failing call in one
    # thread must not overwrite the message another thread is about to read.
    import threading
    null = ctypes.c_void_p(0)
    st = ctypes.create_string_buffer(48)
    stp = ctypes.cast(st, ctypes.c_void_p)
    barrier = threading.Barrier(2)
    seen = {}

    def logprob_thread():
        for _ in range(200):
            assert L.occ_token_logprob(null, 0, 4, 0, 0, null, null, null, null) == 1
            barrier.wait()
            msg = L.occ_last_error()
            barrier.wait()
            seen.setdefault("logprob", set()).add(msg)

    def ewma_thread():
        for _ in range(200):
            assert L.occ_ewma_update(null, null, 0, 1.5, stp, null, 0.9, 1, 0, null) == 1
            barrier.wait()
            msg = L.occ_last_error()
            barrier.wait()
            seen.setdefault("ewma", set()).add(msg)

    ts = [threading.Thread(target=logprob_thread), threading.Thread(target=ewma_thread)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    assert len(seen["logprob"]) == 1 and b"V >= 1" in next(iter(seen["logprob"]))
    assert len(seen["ewma"]) == 1 and b"beta" in next(iter(seen["ewma"]))


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    # without libocc.so every entry point raises; nothing falls back to a CPU path
    import torch
    monkeypatch.setattr(occ, "LIB_PATH", str(tmp_path / "libocc.so"))
    monkeypatch.setattr(occ, "_lib", None)
    with pytest.raises(occ.OccError, match="not built"):
        occ.lib()
    with pytest.raises(occ.OccError):
        occ.occ_loss_workspace_bytes(16, 32)
    if torch.cuda.is_available():
        with pytest.raises(occ.OccError, match="not built"):
            occ.occ_token_logprob(torch.zeros(2, 4, device="cuda"),
                                  torch.zeros(2, dtype=torch.int32, device="cuda"))


def test_concurrent_builds_take_turns():
    # ranks of one job (or parallel test workers) may all call build(): one
    # forced rebuild and two plain ones at the same time must all succeed and
    # leave a library that exports every entry point
    import subprocess
    import sys
    code = "from paper_2605_12070_gb300 import build; build.build(force={})"
    procs = [subprocess.Popen([sys.executable, "-c", code.format(f)], cwd=ROOT,
                              stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True)
             for f in (True, False, False)]
    for p in procs:
        out, err = p.communicate(timeout=900)
        assert p.returncode == 0, err[-2000:]
    L2 = ctypes.CDLL(build.LIB)
    for name in occ.EXPORTS:
        assert hasattr(L2, name), name


def test_options_are_explicit_and_checked(L):
    # the library reads no environment variable: an option changes only through
    # occ_set_option, rejects values it does not know, and -1 restores the default
    import os
    assert "getenv" not in open(os.path.join(os.path.dirname(occ.LIB_PATH), "csrc",
                                             "occ_loss.cu")).read()
    for name, code in occ.OPTIONS.items():
        assert L.occ_get_option(code) == -1, name
    assert L.occ_set_option(2, 256) == 0 and L.occ_get_option(2) == 256
    assert L.occ_set_option(2, 300) == 1 and L.occ_get_option(2) == 256
    assert L.occ_set_option(2, -1) == 0 and L.occ_get_option(2) == -1
    assert L.occ_set_option(99, 1) == 1 and L.occ_get_option(99) == -1
    with occ.options(fused_threads=256, fused_head_bytes=4096):
        assert occ.get_option("fused_threads") == 256 and occ.get_option("fused_head_bytes") == 4096
    assert occ.get_option("fused_threads") == -1 and occ.get_option("fused_head_bytes") == -1
