"""Several GPUs: one process per GPU, each with its own key replica.

Ciphertexts are independent, so a batch shards with no data-path collective:
each rank bootstraps a contiguous slice of the batch through its own
Context.  The only communication is host-side bookkeeping: the maximum of
the per-rank step times (for throughput) and, when a caller wants the whole
result on one rank, a gather of the output slices.
"""

from __future__ import annotations

import numpy as np


def shard_range(total: int, world: int, rank: int) -> tuple[int, int]:
    """(start, count) of rank's contiguous slice; sizes differ by at most one."""
    if world <= 0 or not 0 <= rank < world:
        raise ValueError("bad world/rank")
    base, extra = divmod(total, world)
    start = rank * base + min(rank, extra)
    return start, base + (1 if rank < extra else 0)


def max_over_ranks(value: float, dist=None, device=None) -> float:
    """Largest `value` over all ranks (the slowest rank bounds a step)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(value)
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def gather_rows(local: np.ndarray, total: int, dist=None, dst: int = 0):
    """Concatenate every rank's rows (in rank order) on rank `dst`; other
    ranks get None.  Slices may differ in length by one row."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return local
    import torch
    world, rank = dist.get_world_size(), dist.get_rank()
    width = local.shape[1]
    rows = shard_range(total, world, 0)[1]          # the largest slice
    buf = np.zeros((rows, width), dtype=np.uint64)
    buf[:local.shape[0]] = local
    t = torch.from_numpy(buf.view(np.int64))
    parts = [torch.empty_like(t) for _ in range(world)] if rank == dst else None
    dist.gather(t, parts, dst=dst)
    if rank != dst:
        return None
    out = [parts[r].numpy().view(np.uint64)[:shard_range(total, world, r)[1]] for r in range(world)]
    return np.concatenate(out, axis=0)


def pbs_batch_sharded(ctx, lwe_all: np.ndarray, lut: np.ndarray, dist=None, dst: int = 0):
    """Bootstrap this rank's slice of `lwe_all` with `ctx` and gather all
    outputs on rank `dst` (None elsewhere)."""
    world = dist.get_world_size() if dist is not None and dist.is_initialized() else 1
    rank = dist.get_rank() if world > 1 else 0
    start, count = shard_range(lwe_all.shape[0], world, rank)
    local_in = np.ascontiguousarray(lwe_all[start:start + count])
    local_out = np.zeros((count, lwe_all.shape[1]), dtype=np.uint64)
    if count:
        ctx.pbs_batch(local_in, lut, local_out)
    return gather_rows(local_out, lwe_all.shape[0], dist, dst)
