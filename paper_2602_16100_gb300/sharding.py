"""Data-parallel sharding of the compliance-checking batch across ranks.

Every unit of the path is independent of the others: an intent's selector
row, its pods' placement, its probes' walks and its verdict read only that
intent's inputs plus the shared cluster labels and flow tables (Sec. 4.2, the
per-intent cross-layer check; Sec. 5.5, one verdict per intent).  A batch
therefore splits into contiguous intent ranges with no exchange between
ranks: each rank loads the shared cluster and network, runs its own range on
its own GPU, and the only collectives are host-side bookkeeping outside the
data path: a barrier, the max over ranks of the timed region, and the sum
over ranks of the per-status counters and verdict counts once the batch is
done.

This module holds the host-side range arithmetic, the slicing of an
end-to-end batch and the rank bookkeeping.  It does no compliance arithmetic.
"""
from __future__ import annotations

import dataclasses
from typing import Optional, Tuple

import numpy as np

from . import workloads as W


def shard_range(n_units: int, rank: int, world: int) -> Tuple[int, int]:
    """Contiguous [lo, hi) of `n_units` for `rank` of `world`; the ranges
    cover 0..n_units exactly once and differ in length by at most one."""
    if world < 1 or not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world of {world}")
    if n_units < 0:
        raise ValueError("negative unit count")
    return (n_units * rank) // world, (n_units * (rank + 1)) // world


def shard_seed(base_seed: int, rank: int) -> int:
    """Seed of rank `rank`'s own batch under weak scaling: every rank draws a
    different batch of the same shape, rank 0 the unsharded one."""
    return int(base_seed) + int(rank)


def shard_end_to_end(e: W.EndToEnd, rank: int, world: int) -> W.EndToEnd:
    """The intents [lo, hi) of an end-to-end batch as a batch of their own:
    their selector rows (offsets rebased), placement draws and probes; the
    cluster and the network are shared, not copied."""
    lo, hi = shard_range(e.intents.num_pods, rank, world)
    offs = e.intents.expr_offs
    e0, e1 = int(offs[lo]), int(offs[hi])
    pods, ppg = e.pods_per_intent, e.probes_per_intent
    sel = W.Selectors(hi - lo, (offs[lo:hi + 1] - offs[lo]).astype(np.uint32), e.intents.exprs[e0:e1].copy(), None)
    probes = W.Probes(e.probes.probes[lo * ppg:hi * ppg].copy(), e.probes.hop_cap)
    return dataclasses.replace(e, intents=sel, intent_mask=e.intent_mask[lo:hi].copy(),
                               place_draws=e.place_draws[lo * pods:hi * pods].copy(), probes=probes)


def world_info() -> Tuple[int, int, int]:
    """(rank, world size, local rank) from the launcher's environment."""
    import os
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")),
            int(os.environ.get("LOCAL_RANK", "0")))


def max_over_ranks(x: float, dist=None, device: Optional[str] = None) -> float:
    """Maximum of a host scalar over all ranks (identity without a process
    group).  `device` is where the reduction tensor lives: "cuda" under NCCL,
    "cpu" under gloo."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: int, dist=None, device: Optional[str] = None) -> int:
    """Sum of a host integer over all ranks (identity without a process group)."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return int(x)
    import torch
    t = torch.tensor([int(x)], dtype=torch.int64, device=device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return int(t.item())


def sum_vector_over_ranks(v, dist=None, device: Optional[str] = None) -> np.ndarray:
    """Elementwise sum of an integer vector (per-status counters, verdict
    counts) over all ranks; a copy of `v` without a process group."""
    a = np.asarray(v, dtype=np.int64).copy()
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return a
    import torch
    t = torch.from_numpy(a).to(device or "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return t.cpu().numpy()
