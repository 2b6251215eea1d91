"""Data-parallel plumbing around the occ kernels (torch.distributed).

Tokens are independent, so a global batch shards by rows with no collective
on the data path.  Two small exchanges keep the shards equivalent to one
batch:
  * the token-mean denominator N is the global count of valid tokens (R7); it
    is summed once per batch and passed to every rank as ``denom``, so each
    rank's loss and gradient are already divided by the global N;
  * the EWMA auto-reset (Sec. 5.2) must see the global Train-Infer Mask value
    rho = n_active / n_valid, otherwise ranks would reset their proximal
    parameters at different steps.  ``allreduce_loss_stats`` sums the loss
    and the counters of the device statistics in place (40 bytes), before
    occ_ewma_update reads them.
"""

import torch
import torch.distributed as dist

# word offsets inside occ_loss_stats (include/occ.h)
_F64_LOSS = slice(0, 2)        # loss_sum, loss
_I64_COUNTS = slice(2, 6)      # n_valid, n_rd_out, n_clipped, n_active
_I32_ERR = slice(14, 15)       # err


def global_token_count(n_local, group=None):
    """Sum of the ranks' valid-token counts (host integer)."""
    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() and \
        dist.get_backend(group) == "nccl" else torch.device("cpu")
    t = torch.tensor([int(n_local)], dtype=torch.int64, device=dev)
    dist.all_reduce(t, group=group)
    return int(t.item())


def _allreduce_bits_or(word, group=None):
    """Bitwise OR of a 32-bit word over ranks, in place.  NCCL has no bitwise
    reduction, so each bit becomes a 0/1 indicator, the indicators are
    MAX-reduced, and the word is rebuilt: bit k is set iff some rank set it."""
    shifts = torch.arange(32, dtype=torch.int64, device=word.device)
    bits = (word.to(torch.int64) >> shifts) & 1
    dist.all_reduce(bits, op=dist.ReduceOp.MAX, group=group)
    packed = (bits << shifts).sum()
    word.copy_(torch.where(packed >= 2 ** 31, packed - 2 ** 32, packed).to(torch.int32).view(1))


def allreduce_loss_stats(stats, group=None):
    """In-place sum of loss_sum, loss and the four counters over ranks; the
    err bits are OR-ed (a bit set on any rank is set in the result).
    ``denom`` is left as is: every rank must have used the same global
    denominator."""
    if stats.dtype != torch.uint8 or stats.numel() != 64:
        raise ValueError("stats must be the 64-byte occ_loss_stats tensor")
    f64 = stats.view(torch.float64)
    i64 = stats.view(torch.int64)
    i32 = stats.view(torch.int32)
    dist.all_reduce(f64[_F64_LOSS], group=group)
    dist.all_reduce(i64[_I64_COUNTS], group=group)
    _allreduce_bits_or(i32[_I32_ERR], group=group)
    return stats
