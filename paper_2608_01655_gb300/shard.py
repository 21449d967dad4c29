"""Splitting the order-diverse starts of one plan across processes.

The starts of Algorithm 1 are independent chains: each runs its own greedy
pass and refinement and yields one candidate.  With P processes (one per
GPU), process `rank` runs the starts s with s % P == rank and keeps its best
candidate; the plan's result is then the candidate with the highest
objective, ties to the lowest start index (the same rule as one process).
The only exchange is that final choice: every rank contributes
(objective, start index), all agree on the winner, and the winner's rank
broadcasts its placement.  No data moves between ranks while they plan.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


def my_starts(n_starts: int, rank: int, world: int) -> np.ndarray:
    """Global start indices this rank plans (round-robin)."""
    return np.arange(rank, n_starts, world, dtype=np.int64)


def total_starts(S: int, world: int, scaling: str) -> int:
    """Starts of the whole job: weak scaling plans S starts per process
    (S * world in all), strong scaling splits the S starts of one plan."""
    if scaling not in ("weak", "strong"):
        raise ValueError("scaling must be 'weak' or 'strong'")
    return S * world if scaling == "weak" else S


def rank_orders(default_orders, S: int, rank: int, world: int, scaling: str):
    """The start orders this rank plans and their global start indices.

    default_orders(total) -> [total][W] int32 must give the same orders on
    every rank (pp_default_orders does: it depends on the instance only)."""
    total = total_starts(S, world, scaling)
    orders = np.asarray(default_orders(total), np.int32)
    idx = my_starts(total, rank, world)
    return orders[idx], idx


@dataclass
class ShardResult:
    objective: int
    best_start: int          # global start index of the winner
    placement: np.ndarray    # [W][n] uint8, identical on every rank


def choose_winner(objectives, starts):
    """Highest objective, ties to the lowest global start index."""
    best = None
    for obj, s in zip(objectives, starts):
        if s < 0:
            continue
        if best is None or obj > best[0] or (obj == best[0] and s < best[1]):
            best = (int(obj), int(s))
    return best


def exchange(local_obj: int, local_start: int, placement: np.ndarray, group=None) -> ShardResult:
    """All ranks agree on the best (objective, start) and receive its placement.

    A rank with no start passes local_start = -1.  Uses torch.distributed
    (gloo or NCCL; with NCCL the tensors live on the current CUDA device)."""
    import torch
    import torch.distributed as dist

    world = dist.get_world_size(group)
    backend = dist.get_backend(group)
    dev = torch.device("cuda", torch.cuda.current_device()) if backend == "nccl" else torch.device("cpu")
    mine = torch.tensor([int(local_obj), int(local_start)], dtype=torch.int64, device=dev)
    allv = [torch.zeros(2, dtype=torch.int64, device=dev) for _ in range(world)]
    dist.all_gather(allv, mine, group=group)
    pairs = [(int(v[0].item()), int(v[1].item())) for v in allv]
    obj, start = choose_winner([p[0] for p in pairs], [p[1] for p in pairs])
    owner = [r for r, p in enumerate(pairs) if p == (obj, start)][0]
    buf = torch.from_numpy(np.ascontiguousarray(placement, dtype=np.uint8)).to(dev)
    dist.broadcast(buf, src=owner, group=group)
    return ShardResult(obj, start, buf.cpu().numpy())


def plan_sharded(run_starts, orders: np.ndarray, n_shape, rank: int, world: int, group=None) -> ShardResult:
    """Run this rank's share of the starts and exchange the winner.

    run_starts(sub_orders) -> (per_start_objective, best_local_index, placement)
    plans the given start orders (rows of `orders`) on this rank's device."""
    idx = my_starts(orders.shape[0], rank, world)
    if idx.size:
        per, best_local, placement = run_starts(orders[idx])
        obj, start = int(per[best_local]), int(idx[best_local])
    else:
        obj, start, placement = 0, -1, np.zeros(n_shape, np.uint8)
    return exchange(obj, start, placement, group)
