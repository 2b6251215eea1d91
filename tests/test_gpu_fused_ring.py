"""The persistent TMA-ring fused kernel (OCC_FUSED_VARIANT=ring) against the oracle.

The default fused kernel is the two-pass L2 kernel; the ring kernel (one
persistent CTA per SM, cp.async.bulk copies into a shared-memory head and an
mbarrier-guarded ring, tokens fetched from a device counter) is kept as a
tuning alternative.  The variant is read once per process, so the fused
parity tests run again in a child process with it selected (their
diagnostics cases keep the default kernel, which the ring variant leaves to
it).
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_fused_parity_suite_with_the_ring_kernel():
    env = dict(os.environ, OCC_FUSED_VARIANT="ring")
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_fused.py"),
                        os.path.join(ROOT, "tests", "test_gpu_graph.py"),
                        os.path.join(ROOT, "tests", "test_gpu_pipeline.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert " passed" in r.stdout
