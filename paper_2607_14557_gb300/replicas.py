"""Multi-GPU plumbing of the hot path: independent replicas, no data-path collective.

Sequences are independent through detection, compaction and every layer, so
N GPUs run N independent problems; the only cross-rank traffic is timing and
counting at the host level (a barrier, the maximum of the per-rank step times,
the sum of the per-rank token counts).  ``shard_sequences`` splits one batch
across ranks by tokens (longest first onto the least-loaded rank) for callers
that serve a single batch on several GPUs.
"""
from __future__ import annotations

from typing import List, Sequence

import torch
import torch.distributed as dist


def shard_sequences(token_counts: Sequence[int], world: int) -> List[List[int]]:
    """Greedy token-balanced assignment: sequences in decreasing token count,
    each to the rank with the fewest tokens so far (ties: lowest rank; equal
    counts keep batch order).  Returns, per rank, its sequence indices in
    increasing order."""
    if world < 1:
        raise ValueError("world must be >= 1")
    order = sorted(range(len(token_counts)), key=lambda i: (-int(token_counts[i]), i))
    load = [0] * world
    parts: List[List[int]] = [[] for _ in range(world)]
    for i in order:
        r = min(range(world), key=lambda k: (load[k], k))
        parts[r].append(i)
        load[r] += int(token_counts[i])
    return [sorted(p) for p in parts]


def _reduce(value: float, op, device) -> float:
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=op)
    return float(t.item())


def max_over_ranks(value: float, device=None) -> float:
    """Maximum of ``value`` over the ranks of the default process group (the
    value itself when no group is initialised)."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    return _reduce(value, dist.ReduceOp.MAX, device)


def sum_over_ranks(value: float, device=None) -> float:
    """Sum of ``value`` over the ranks of the default process group."""
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    return _reduce(value, dist.ReduceOp.SUM, device)


def barrier(device=None) -> None:
    """Process-group barrier (when one exists), then a device synchronise
    when ``device`` is a CUDA device."""
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()
    if device is not None and torch.device(device).type == "cuda":
        torch.cuda.synchronize(device)
