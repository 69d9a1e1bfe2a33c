"""Host-side planning for runs on several GPUs (one process per GPU).

Every selection unit of the per-tensor and per-block scopes is a whole tensor
or a tile of one, so a parameter set splits across GPUs by whole tensors with
no collective on the data path: each rank updates or merges its own tensors.
Only the timing needs the ranks together (the step time of a run is the
slowest rank's).  The global scope, one unit over all tensors, would need a
histogram all-reduce per radix level and is not split here.
"""
from __future__ import annotations

from typing import List, Sequence


def shard_tensors(numels: Sequence[int], world: int) -> List[List[int]]:
    """Assign tensors to `world` ranks, balancing entries: largest tensor
    first, each to the rank with the fewest entries so far (ties to the lower
    rank).  Deterministic; every tensor goes to exactly one rank; a rank's
    list keeps the tensors' original order."""
    if world < 1:
        raise ValueError("world must be >= 1")
    load = [0] * world
    owner = [0] * len(numels)
    for q in sorted(range(len(numels)), key=lambda i: (-int(numels[i]), i)):
        r = min(range(world), key=lambda j: (load[j], j))
        owner[q] = r
        load[r] += int(numels[q])
    return [[q for q in range(len(numels)) if owner[q] == r] for r in range(world)]


def reduce_step_ms(ms: float, device=None) -> float:
    """The step time over all ranks of the default process group: the
    maximum.  Without a group (one process) the value itself."""
    import torch
    import torch.distributed as dist
    if not dist.is_available() or not dist.is_initialized() or dist.get_world_size() == 1:
        return float(ms)
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(params_all_ranks: int, ms: float) -> float:
    """Whole-job parameters per second, in G params/s, for a step time of ms."""
    return params_all_ranks / (ms * 1e-3) / 1e9
