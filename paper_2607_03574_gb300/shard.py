"""Partition of one lane population across processes (one process per GPU).

Lanes are independent (section 6, multicore execution: candidates in a population
share no mutable state), so a population of B lanes splits into contiguous slices, one
per rank, with no exchange during the replay: every rank replays its slice with the
same tape and writes its own slice of loss and gradient.  The only communication is a
host-side gather of the slices onto rank 0 after the replay.

Host logic only (numpy and torch.distributed on CPU tensors); nothing here computes
any part of the replay.
"""
from __future__ import annotations

import numpy as np


def lane_slice(B: int, world: int, rank: int) -> tuple[int, int]:
    """Half-open lane range [lo, hi) owned by `rank` among `world` ranks.

    Contiguous and balanced: the first B mod world ranks own one lane more than the
    others; the slices are disjoint and cover [0, B) in rank order."""
    if world < 1 or not 0 <= rank < world or B < 0:
        raise ValueError(f"bad partition arguments B={B} world={world} rank={rank}")
    base, extra = divmod(B, world)
    lo = rank * base + min(rank, extra)
    return lo, lo + base + (1 if rank < extra else 0)


def gather_lanes(local: np.ndarray, B: int, world: int, rank: int, group=None):
    """Gather every rank's slice of a per-lane array (leading axis = lanes) onto rank 0.

    `local` holds this rank's lanes lane_slice(B, world, rank).  Rank 0 returns the
    (B, ...) array in lane order; the other ranks return None.  Slices are padded to a
    common length for the collective and trimmed again on rank 0.  Runs over the
    process group `group` (a CPU-capable backend such as gloo)."""
    import torch
    import torch.distributed as dist

    local = np.ascontiguousarray(local)
    lo, hi = lane_slice(B, world, rank)
    if local.shape[0] != hi - lo:
        raise ValueError(f"rank {rank} holds {local.shape[0]} lanes, its slice has {hi - lo}")
    if world == 1:
        return local.copy()
    rows = -(-B // world)
    pad = np.zeros((rows,) + local.shape[1:], dtype=local.dtype)
    pad[: hi - lo] = local
    t = torch.from_numpy(pad)
    bufs = [torch.empty_like(t) for _ in range(world)] if rank == 0 else None
    dist.gather(t, gather_list=bufs, dst=0, group=group)
    if rank != 0:
        return None
    out = np.empty((B,) + local.shape[1:], dtype=local.dtype)
    for r in range(world):
        a, b = lane_slice(B, world, r)
        out[a:b] = bufs[r].numpy()[: b - a]
    return out
