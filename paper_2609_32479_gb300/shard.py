"""Host-side sharding of a track batch across ranks (replicas; no exchange step).

Tracks are independent (Sec. 4), so a multi-GPU run gives each rank a
contiguous slice of the batch and, where one host needs all results, gathers
the [B, 5] outputs.  These helpers hold only index arithmetic and the gather;
the per-rank compute is the caller's (the C-ABI forward on its own GPU)."""
from __future__ import annotations

from typing import Tuple

import numpy as np


def shard_range(n_tracks: int, rank: int, world: int) -> Tuple[int, int]:
    """Contiguous [begin, end) slice of rank `rank`; sizes differ by at most one."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError("bad rank/world")
    base, extra = divmod(n_tracks, world)
    begin = rank * base + min(rank, extra)
    return begin, begin + base + (1 if rank < extra else 0)


def gather_outputs(local: np.ndarray, n_tracks: int, group=None) -> np.ndarray:
    """All-gather the per-rank [n_r, 5] outputs into [n_tracks, 5] in track order
    (torch.distributed; any backend).  Every rank receives the full array."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    rank = dist.get_rank(group)
    b, e = shard_range(n_tracks, rank, world)
    if local.shape[0] != e - b:
        raise ValueError("local output does not match this rank's shard")
    width = max(shard_range(n_tracks, r, world)[1] - shard_range(n_tracks, r, world)[0] for r in range(world))
    pad = np.zeros((width, local.shape[1]), dtype=local.dtype)
    pad[:local.shape[0]] = local
    parts = [torch.zeros_like(torch.from_numpy(pad)) for _ in range(world)]
    dist.all_gather(parts, torch.from_numpy(pad), group=group)
    out = np.empty((n_tracks, local.shape[1]), dtype=local.dtype)
    for r in range(world):
        rb, re = shard_range(n_tracks, r, world)
        out[rb:re] = parts[r].numpy()[:re - rb]
    return out
