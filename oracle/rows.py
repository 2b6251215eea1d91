"""Row-chunk driver for running the oracle over large batches.

TEST INFRASTRUCTURE ONLY.  Holds no arithmetic of the method: it cuts a
(T, V) tensor into row chunks, upcasts each chunk exactly to float64 and runs
a caller-supplied oracle function on it, optionally on a thread pool.  numpy
releases the GIL inside its array loops, so threads give real parallelism and
avoid forking a process that may hold a CUDA context.
"""

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np


def host_cores():
    """Cores this process may run on (the figure reported beside CPU timings)."""
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def to_f64(x):
    """Exact float64 copy of a host tensor/array chunk (bf16 and fp32 upcast exactly)."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return x.detach().to("cpu").to(torch.float64).numpy()
    except ImportError:  # pragma: no cover
        pass
    return np.asarray(x, dtype=np.float64)


def map_row_chunks(fn, rows, chunk=64, threads=None):
    """Apply ``fn(row_index_array)`` to consecutive chunks of ``rows``.

    Returns the list of results in chunk order (the order does not depend on
    the thread count).
    """
    rows = np.asarray(rows)
    pieces = [rows[i:i + chunk] for i in range(0, rows.size, chunk)]
    threads = threads or host_cores()
    if threads <= 1 or len(pieces) <= 1:
        return [fn(p) for p in pieces]
    with ThreadPoolExecutor(max_workers=threads) as ex:
        return list(ex.map(fn, pieces))
