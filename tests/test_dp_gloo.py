"""World-size-2 tests of the data-parallel plumbing on CPU (gloo).

The token-parallel design: ranks hold disjoint row shards of one batch, use
the global valid-token count as the token-mean denominator, and all-reduce
the loss statistics before the EWMA reset decision.  Here each rank's kernel
results are stood in for by the oracle on its shard (no GPU on this
machine); the checks are that the reduced statistics equal the unsharded
batch's and that both ranks take the same reset decision.
"""

import os
import socket
import struct

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2605_12070_gb300 import dp, occ


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _stats_bytes(o, denom, err=0):
    raw = struct.pack("<2d5q2i", o["loss_sum"], o["loss_sum"] / denom, o["n_valid"],
                      o["n_rd_out"], o["n_clipped"], o["n_active"], denom, err, 0)
    return torch.frombuffer(bytearray(raw), dtype=torch.uint8).clone()


def _batch(seed=0, T=96, V=50):
    rng = np.random.default_rng(seed)
    z = rng.normal(0, 2, size=(T, V))
    zo = z + rng.normal(0, 0.4, size=(T, V))
    ids = rng.integers(0, V, size=T)
    lo, _ = oracle.token_logprob(zo, ids)
    lmu = lo + rng.normal(0, 0.3, size=T)
    adv = rng.normal(0, 1, size=T)
    mask = (rng.random(T) < 0.8).astype(np.uint8)
    return z, ids, lo, lmu, adv, mask


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        z, ids, lo, lmu, adv, mask = _batch()
        T = len(ids)
        p = oracle.LossParams(0.7, 1.4, 0.2, 0.28)
        rows = np.arange(rank, T, world)                   # this rank's shard
        n_local = int(mask[rows].sum())
        N = dp.global_token_count(n_local)
        lt, _ = oracle.token_logprob(z[rows], ids[rows])
        o = oracle.token_terms(lt, lo[rows], lmu[rows], adv[rows], mask[rows], p, N=N)
        # rank 0 reports a dropped id, rank 1 two other bits (one the sign bit):
        # the reduced word must keep every bit (OR), which MAX would not
        err = occ.DATA_ERR_BAD_ID if rank == 0 else (2 | -2 ** 31)
        stats = _stats_bytes(o, N, err=err)
        dp.allreduce_loss_stats(stats)
        s = occ.decode_loss_stats(stats)
        _, _, reset, _ = oracle.ewma_coefficients(oracle.EwmaState(w=3.0), 0.75,
                                                  n_active=s.n_active, n_valid=s.n_valid,
                                                  tau=0.9)
        q.put((rank, N, s, reset))
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_sharded_batch_equals_unsharded():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for pr in procs:
        pr.start()
    res = sorted([q.get(timeout=100) for _ in range(world)], key=lambda r: r[0])
    for pr in procs:
        pr.join(timeout=30)
        assert pr.exitcode == 0
    z, ids, lo, lmu, adv, mask = _batch()
    p = oracle.LossParams(0.7, 1.4, 0.2, 0.28)
    lt, _ = oracle.token_logprob(z, ids)
    ref = oracle.token_terms(lt, lo, lmu, adv, mask, p)
    _, _, ref_reset, _ = oracle.ewma_coefficients(oracle.EwmaState(w=3.0), 0.75,
                                                  n_active=ref["n_active"],
                                                  n_valid=ref["n_valid"], tau=0.9)
    for rank, N, s, reset in res:
        assert N == ref["N"]
        assert (s.n_valid, s.n_rd_out, s.n_clipped, s.n_active) == (
            ref["n_valid"], ref["n_rd_out"], ref["n_clipped"], ref["n_active"])
        assert abs(s.loss - ref["loss"]) < 1e-12 and abs(s.loss_sum - ref["loss_sum"]) < 1e-12
        assert s.denom == ref["N"]
        assert s.err == (occ.DATA_ERR_BAD_ID | 2 | -2 ** 31)
        assert reset == ref_reset
    assert res[0][3] == res[1][3]
