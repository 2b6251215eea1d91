"""Runs the float64 oracle on (sampled rows of) a GPU batch, for the parity tests.

Test infrastructure: rows are copied to the host chunk by chunk, upcast
exactly to float64 and evaluated with ``oracle`` on a thread pool.
"""

import numpy as np
import torch

from oracle import LossParams, softmax_grad_rows, token_logprob, token_terms
from oracle.rows import map_row_chunks, to_f64


def logprob_rows(z, ids, rows, chunk=32):
    """Oracle R1 for the given rows of a device logits tensor: (logp, lse) float64."""
    rows = np.asarray(rows, dtype=np.int64)
    ids_h = ids.to("cpu").numpy().astype(np.int64)

    def fn(r):
        zr = to_f64(z[torch.as_tensor(r, device=z.device)])
        return token_logprob(zr, ids_h[r])

    parts = map_row_chunks(fn, rows, chunk=chunk)
    if not parts:
        return np.zeros(0), np.zeros(0)
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def loss_params(batch, **kw):
    d = batch.thresholds()
    d.update(kw)
    return LossParams(**d)


def oracle_loss(batch, logp_theta, logp_old, params, N=None):
    """Oracle R2..R9 on full per-token arrays (logp_theta may be NaN on masked rows)."""
    ids = batch.ids.to("cpu").numpy().astype(np.int64)
    mask = None if batch.mask is None else batch.mask.to("cpu").numpy()
    id_ok = (ids >= 0) & (ids < batch.V)
    return token_terms(np.nan_to_num(logp_theta), logp_old, batch.logp_mu.to("cpu").numpy(),
                       batch.adv.to("cpu").numpy(), mask, params, id_ok=id_ok, N=N)


def dlogits_rows(batch, rows, lse, g, chunk=32):
    """Oracle R8 rows of dL/dz for the given rows (lse, g indexed like rows)."""
    rows = np.asarray(rows, dtype=np.int64)
    ids_h = batch.ids.to("cpu").numpy().astype(np.int64)
    pos = {int(r): k for k, r in enumerate(rows)}

    def fn(r):
        k = np.array([pos[int(x)] for x in r])
        zr = to_f64(batch.z_theta[torch.as_tensor(r, device=batch.z_theta.device)])
        return softmax_grad_rows(zr, np.clip(ids_h[r], 0, batch.V - 1), lse[k], g[k])

    return np.concatenate(map_row_chunks(fn, rows, chunk=chunk), axis=0)


def fp32(x):
    """The float32 interface type of per-token log-probabilities."""
    return np.asarray(x, dtype=np.float64).astype(np.float32)
