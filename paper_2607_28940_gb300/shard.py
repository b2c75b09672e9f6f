"""Request sharding across GPUs (one process per GPU).

Requests are independent (the per-candidate factorisation of Sec. 4.1.3 and a
separate cache per request), so a batch of world * R requests splits into
contiguous blocks of R requests per rank with no collective on the data path.
Only measurements are reduced across ranks.
"""
from __future__ import annotations

from typing import List

from . import workload as W


def global_workload(per_rank: W.Workload, world: int) -> W.Workload:
    """The whole job: world times the per-rank request count, same seed."""
    return W.with_sizes(per_rank, n_req=per_rank.n_req * world)


def shard_requests(n_per_rank: int, rank: int, world: int) -> List[int]:
    """Requests of `rank` in the global batch: a contiguous block."""
    if not 0 <= rank < world:
        raise ValueError(f"rank {rank} outside world {world}")
    return list(range(rank * n_per_rank, (rank + 1) * n_per_rank))


def reduce_max(value: float, device="cpu") -> float:
    """Max of `value` over all ranks (identity without a process group)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())
