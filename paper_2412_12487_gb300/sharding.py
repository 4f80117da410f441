"""Scenario sharding over several GPUs, one process per GPU.

Every scenario is its own composition of the same graph, so a batch of scenarios
splits into contiguous slices, one per rank, each composed by that rank's own
context with a full copy of the graph.  The data path has no exchange: ranks meet
only to time the step (the slowest rank's time counts) and, when the caller wants
the whole batch's results in one place, to gather them on rank 0 afterwards over
a host (gloo) group.
"""
from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import numpy as np

from . import workloads as W


def shard_bounds(n_total: int, world: int, rank: int) -> Tuple[int, int]:
    """Scenarios [s0, s1) of ``rank``: contiguous slices whose sizes differ by at most one."""
    if world < 1 or not 0 <= rank < world or n_total < 0:
        raise ValueError(f"bad shard request: n_total={n_total} world={world} rank={rank}")
    q, r = divmod(n_total, world)
    s0 = rank * q + min(rank, r)
    return s0, s0 + q + (1 if rank < r else 0)


def slice_scenarios(sc: W.Scenarios, s0: int, s1: int) -> W.Scenarios:
    """Columns [s0, s1) of every per-scenario array of ``sc`` (durations included)."""
    cols = slice(s0, s1)
    return W.Scenarios(
        dur=np.ascontiguousarray(sc.dur[:, cols]),
        alpha_ns=sc.alpha_ns[cols].copy(), bw_intra=sc.bw_intra[cols].copy(),
        lat_intra=sc.lat_intra[cols].copy(), bw_inter=sc.bw_inter[cols].copy(),
        lat_inter=sc.lat_inter[cols].copy(), delta=sc.delta[cols].copy(),
        slowdown=np.ascontiguousarray(sc.slowdown[:, cols]),
        peak_flop_per_ns=sc.peak_flop_per_ns[cols].copy(),
        chunk_max_bytes=sc.chunk_max_bytes, chunk_bytes=sc.chunk_bytes)


def max_over_ranks(values: Sequence[float], group=None, device=None) -> List[float]:
    """Element-wise maximum of ``values`` over the ranks of ``group`` (default: the
    world); the identity without an initialised process group."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()):
        return [float(v) for v in values]
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    return [float(v) for v in t.cpu()]


def gather_scenarios(x: np.ndarray, n_total: int, group=None) -> Optional[np.ndarray]:
    """Concatenates every rank's per-scenario results along the last axis, in
    scenario order, on rank 0 of ``group`` (a gloo group: host memory only).  The
    other ranks get None."""
    import torch
    import torch.distributed as dist
    world = dist.get_world_size(group)
    rank = dist.get_rank(group)
    s0, s1 = shard_bounds(n_total, world, rank)
    if x.shape[-1] != s1 - s0:
        raise ValueError(f"rank {rank} holds {x.shape[-1]} scenarios, expected {s1 - s0}")
    lead = x.shape[:-1]
    width = max(shard_bounds(n_total, world, r)[1] - shard_bounds(n_total, world, r)[0] for r in range(world))
    buf = torch.zeros(lead + (width,), dtype=torch.from_numpy(np.empty(0, dtype=x.dtype)).dtype)
    buf[..., : s1 - s0] = torch.from_numpy(np.ascontiguousarray(x))
    parts = [torch.empty_like(buf) for _ in range(world)] if rank == 0 else None
    dist.gather(buf, parts, dst=dist.get_global_rank(group, 0) if group is not None else 0, group=group)
    if rank != 0:
        return None
    out = []
    for r in range(world):
        a, b = shard_bounds(n_total, world, r)
        out.append(parts[r][..., : b - a].numpy())
    return np.concatenate(out, axis=-1)
