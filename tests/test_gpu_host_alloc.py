"""Huge-page-backed pinned host buffers (occ_host_alloc / occ_host_free).

The buffers are zero-filled, page-locked (device copies are asynchronous),
round-trip through the device bit for bit, serve as the proximal buffer of
occ_ewma_update_host, and are released when their last view is gone.
"""

import gc

import pytest
import torch

from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_ewma_buffers

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("shape,dtype", [((3, 1000003), torch.bfloat16), ((257,), torch.float32),
                                         ((1 << 28,), torch.uint8)])
def test_round_trip_and_zero_fill(shape, dtype):
    h = occ.occ_host_alloc(shape, dtype)
    assert h.shape == torch.Size(shape) and h.dtype == dtype and h.is_pinned()
    assert not torch.any(h.view(torch.uint8))
    src = torch.randint(0, 255, h.view(torch.uint8).shape, dtype=torch.uint8)
    h.view(torch.uint8).copy_(src)
    d = torch.empty_like(h, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        d.copy_(h, non_blocking=True)
    s.synchronize()
    back = occ.occ_host_alloc(shape, dtype)
    back.copy_(d, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(back.view(torch.uint8), src)
    del h, back, d
    gc.collect()


def test_views_keep_the_buffer_alive():
    h = occ.occ_host_alloc((1 << 20,), torch.float32)
    v = h[10:20]
    v.fill_(3.0)
    del h
    gc.collect()
    assert torch.all(v == 3.0)  # the mapping outlives the parent tensor
    d = v.to("cuda", non_blocking=True)
    torch.cuda.synchronize()
    assert torch.all(d == 3.0)


def test_host_buffer_for_the_host_resident_ewma():
    n = 2_000_011
    th, tp = make_ewma_buffers(n, seed=4, device="cuda")
    tp = tp.to(torch.bfloat16)
    host = occ.occ_host_alloc((n,), torch.bfloat16)
    host.copy_(tp.cpu())
    dev = tp.clone()
    st_d = occ.new_ewma_state("cuda", w0=2.0)
    st_h = occ.new_ewma_state("cuda", w0=2.0)
    staging = torch.empty(1 << 20, dtype=torch.uint8, device="cuda")
    for step in range(2):
        occ.occ_ewma_update_bf16(dev, th, 0.8, st_d, sr_seed=31 + step)
        occ.occ_ewma_update_host(host, th, 0.8, st_h, staging, sr_seed=31 + step)
        torch.cuda.synchronize()
        assert torch.equal(host, dev.cpu()), step


def _rss_bytes():
    with open("/proc/self/status") as f:
        return next(int(l.split()[1]) * 1024 for l in f if l.startswith("VmRSS:"))


def test_release_returns_the_mapping():
    # page-locked memory is resident: the process's RSS rises by the buffer and
    # falls back once the last view is gone
    nbytes = 2 << 30
    before = _rss_bytes()
    h = occ.occ_host_alloc((nbytes,), torch.uint8)
    h[::1 << 20] = 1
    held = _rss_bytes()
    assert held - before >= nbytes * 0.9
    del h
    gc.collect()
    after = _rss_bytes()
    assert after - before <= nbytes * 0.1
