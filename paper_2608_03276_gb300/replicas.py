"""Replica bookkeeping for runs on several GPUs of one node.

The compression path partitions into independent (layer, document, KV head)
units with no exchange between them, so N GPUs run N independent replicas
(weak scaling): each rank compresses its own stack of layers, drawn with its
own seed.  The only cross-rank operations are a barrier on each side of the
timed region and the maximum of the per-rank step times; nothing here touches
the data path, and there is no collective on it.
"""
from __future__ import annotations

import os


def dist_env():
    """(rank, world size, local rank) from the launcher's environment."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init(backend: str, timeout_s: float = 600.0) -> None:
    """Joins the replica group.  The timeout bounds every barrier and
    reduction: a rank that died or hung makes the others' next collective
    fail within it instead of blocking them."""
    import datetime
    import torch.distributed as dist
    dist.init_process_group(backend, timeout=datetime.timedelta(seconds=timeout_s))


def rank_seed(seed: int, rank: int) -> int:
    """Seed of rank `rank`'s replica: every rank compresses different data."""
    return seed + 7919 * rank


def barrier() -> None:
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.barrier()


def max_over_ranks(ms: float, device=None) -> float:
    """The slowest rank's step time: the whole job finishes with it."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(ms)
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_value(tokens_per_layer: int, layers: int, world: int, ms: float) -> float:
    """Context tokens compressed per second per layer over all ranks: every
    rank compresses `layers` layers of `tokens_per_layer` tokens per step."""
    return tokens_per_layer * layers * world / (ms / 1e3)
