"""Data-parallel sharding of the chunk-parallel Comba step across ranks.

The recurrence of section 3 couples tokens only within one sequence and one
head, so a batch splits over sequences with no exchange on the data path: every
rank runs ``comba_chunk_fwd``/``comba_chunk_bwd`` on its own sequences.  The
only cross-rank quantities are the gradients of the per-head parameters
``b`` and ``d`` (section 3.1 feedback strength and output correction), which
are sums over all sequences; a data-parallel trainer reduces them with its
other parameter gradients (``reduce_param_grads``).  Host logic only: no CUDA
work is issued here.
"""
from __future__ import annotations

import numpy as np


def shard_bounds(n_units: int, world: int, rank: int) -> tuple[int, int]:
    """Contiguous balanced range [lo, hi) of `n_units` for `rank` of `world` (sizes differ by <= 1)."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world {world}")
    base, extra = divmod(n_units, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def shard_packed(cu_seqlens, world: int, rank: int):
    """Token-balanced split of packed sequences (``cu_seqlens`` int [N+1]).

    Sequences stay whole.  Rank r takes the sequences whose first token lies in
    the r-th equal slice of the token range, so every sequence goes to exactly
    one rank and the ranks' token counts differ by at most one sequence.
    Returns ``(seq_lo, seq_hi, tok_lo, tok_hi, local_cu)`` with ``local_cu``
    rebased to the shard's first token (int64).
    """
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    if cu.ndim != 1 or cu.size < 1 or cu[0] != 0 or np.any(np.diff(cu) < 0):
        raise ValueError("cu_seqlens must be non-decreasing and start at 0")
    if world <= 0 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world {world}")
    total = int(cu[-1])
    starts = cu[:-1]

    def first_seq(r):
        if r >= world:
            return starts.size
        cut = (total * r + world - 1) // world          # ceil(total * r / world)
        return int(np.searchsorted(starts, cut, side="left")) if r > 0 else 0

    s_lo, s_hi = first_seq(rank), first_seq(rank + 1)
    t_lo, t_hi = int(cu[s_lo]), int(cu[s_hi])
    return s_lo, s_hi, t_lo, t_hi, cu[s_lo:s_hi + 1] - t_lo


def rank_seed_offset(rank: int) -> int:
    """Seed offset of a rank's synthetic batch under weak scaling (distinct data per rank)."""
    return 1_000_003 * rank


def reduce_param_grads(grads: dict, dist, keys=("db", "dd")) -> dict:
    """Sum the per-head parameter gradients over ranks in place (the one cross-rank step)."""
    if dist is not None and dist.is_initialized() and dist.get_world_size() > 1:
        for k in keys:
            if grads.get(k) is not None:
                dist.all_reduce(grads[k], op=dist.ReduceOp.SUM)
    return grads


def max_over_ranks(value: float, dist, device=None) -> float:
    """Maximum of a per-rank scalar (e.g. milliseconds per step) over all ranks."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())
