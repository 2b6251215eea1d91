"""The persistent TMA-ring fused kernel (option fused_variant = 1) against the oracle.

The default fused kernel is the two-pass L2 kernel; the ring kernel (one
persistent CTA per SM, cp.async.bulk copies into a shared-memory head and an
mbarrier-guarded ring, tokens fetched from a device counter) is the
alternative.  The fused parity tests, the CUDA-graph tests and the host-fed
pipeline tests run again in a child process that selects it before any test
(their diagnostics cases keep the default kernel, which the ring variant
leaves to it).
"""

import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import sys
sys.path.insert(0, {root!r})
from paper_2605_12070_gb300 import occ
occ.set_option("fused_variant", 1)
import pytest
sys.exit(pytest.main(["-q", "-x", "-p", "no:cacheprovider", *{files!r}]))
"""


def test_fused_parity_suite_with_the_ring_kernel():
    files = [os.path.join(ROOT, "tests", f) for f in
             ("test_gpu_fused.py", "test_gpu_graph.py", "test_gpu_pipeline.py")]
    r = subprocess.run([sys.executable, "-c", CHILD.format(root=ROOT, files=files)],
                       cwd=ROOT, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
    assert " passed" in r.stdout
