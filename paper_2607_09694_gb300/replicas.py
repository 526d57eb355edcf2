"""Host-side helpers for running the depth path on several GPUs of one node.

The mix has no exchange between tokens in the forward pass, and its only
cross-token coupling in the backward pass (dq, a sum over tokens) belongs to
the ordinary data-parallel gradient all-reduce of the query parameters.  This
build therefore runs *replicas*: every rank processes its own token batch on
its own GPU with no data-path collective; the ranks meet only for the timing
barrier and for the max of their elapsed times.
"""
from __future__ import annotations

import os


def init_from_env():
    """(dist module or None, rank, local_rank, world_size) from torchrun's
    environment; creates the process group (nccl with CUDA, else gloo) for N > 1."""
    import torch
    import torch.distributed as dist

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1 and not dist.is_initialized():
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    return (dist if world > 1 else None), rank, local, world


def max_over_ranks(dist, value: float, device=None) -> float:
    """The largest `value` over all ranks (the slowest rank's time)."""
    if dist is None:
        return float(value)
    import torch

    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def token_range(T: int, rank: int, world: int) -> tuple[int, int]:
    """Contiguous share [start, stop) of T tokens for `rank` when one batch is split
    across ranks instead of replicated (shares differ by at most one token)."""
    if world < 1 or not 0 <= rank < world or T < 0:
        raise ValueError("need 0 <= rank < world and T >= 0")
    base, extra = divmod(T, world)
    start = rank * base + min(rank, extra)
    return start, start + base + (1 if rank < extra else 0)
