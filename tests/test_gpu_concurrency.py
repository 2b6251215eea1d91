"""Calls from several host threads on separate streams.

The library keeps no per-call host state beyond thread-local error messages
and once-per-process caches (SM count, kernel attributes), so concurrent
calls on different streams, each with its own workspace and outputs, must
give the results of the same calls made one after another.
"""

import threading

import pytest
import torch

from paper_2605_12070_gb300 import occ
from paper_2605_12070_gb300.workloads import make_ewma_buffers, make_loss_batch

pytestmark = pytest.mark.gpu


def _step(b, th, tp, st, stream=None):
    out = occ.occ_decoupled_loss_fused(b.z_theta, b.z_old, b.ids, b.logp_mu, b.adv, b.mask,
                                       **b.thresholds(), stream=stream)
    occ.occ_ewma_update(tp, th, 0.9, st, stats=out["stats"], tau=0.5, stream=stream)
    return out


def test_threads_on_separate_streams_match_sequential_calls():
    n_threads, steps = 4, 3
    batches = [make_loss_batch("agentic_bf16_v151936", T=256, seed=60 + k, device="cuda")
               for k in range(n_threads)]
    ewma = [make_ewma_buffers(500_009, seed=60 + k, device="cuda") for k in range(n_threads)]
    # sequential reference
    ref = []
    for b, (th, tp0) in zip(batches, ewma):
        tp, st = tp0.clone(), occ.new_ewma_state("cuda", w0=2.0)
        for _ in range(steps):
            out = _step(b, th, tp, st)
        ref.append((out, tp, st))
    torch.cuda.synchronize()
    # concurrent: one host thread and one stream per batch
    got = [None] * n_threads
    errors = []
    start = threading.Barrier(n_threads)

    def worker(k):
        try:
            s = torch.cuda.Stream()
            th, tp0 = ewma[k]
            with torch.cuda.stream(s):
                tp, st = tp0.clone(), occ.new_ewma_state("cuda", w0=2.0, stream=s)
                start.wait()
                for _ in range(steps):
                    out = _step(batches[k], th, tp, st, stream=s)
            s.synchronize()
            got[k] = (out, tp, st)
        except Exception as e:  # surfaced below
            errors.append(e)

    ts = [threading.Thread(target=worker, args=(k,)) for k in range(n_threads)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    assert not errors, errors
    torch.cuda.synchronize()
    for (o_ref, tp_ref, st_ref), (o, tp, st) in zip(ref, got):
        for key in ("stats", "dlogits", "logp", "logp_old", "flags"):
            assert torch.equal(o[key], o_ref[key]), key
        assert torch.equal(tp, tp_ref) and torch.equal(st, st_ref)
