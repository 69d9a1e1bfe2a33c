"""Host-side planning for runs on several GPUs (one process per GPU).

Every selection unit of the per-tensor and per-block scopes is a whole tensor
or a tile of one, so a parameter set splits across GPUs by whole tensors with
no collective on the data path: each rank updates or merges its own tensors.
Only the timing needs the ranks together (the step time of a run is the
slowest rank's).

A unit split over ranks -- one huge tensor cut into element ranges, or the
global scope over tensors spread across ranks -- has a real exchange step:
``split_unit_select`` finds the unit's exact threshold with one all-reduce of
the ranks' digit histograms per radix level, then an all-gather of the ranks'
tie counts, so that every rank keeps its share of the ties at the threshold
lowest position first (App. F TopKMask with the lowest-index tie rule).
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Callable, List, Sequence


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


# radix digits of the 31-bit magnitude key (|tau| as binary32 bits, sign cleared)
_DIGITS = (11, 11, 9)


@dataclass
class SplitSelect:
    """The exact selection of one unit split over ranks, as one rank sees it.

    k, t, count_above, ties_at_thresh and ties_taken describe the whole unit
    (t = 0xFFFFFFFF when k = 0); ``take`` is how many of this rank's entries
    with key == t are kept, lowest local position first.  A rank keeps the
    entries with key > t and its first ``take`` entries with key == t."""
    k: int
    t: int
    count_above: int
    ties_at_thresh: int
    ties_taken: int
    take: int


def split_unit_select(n_local: int, density: float,
                      local_hist: Callable[[int, int, int, int], Sequence[int]],
                      local_ties: Callable[[int], int], group=None) -> SplitSelect:
    """Exact TopKMask of one selection unit whose entries are split over the
    ranks of ``group`` in rank order (rank r's positions precede rank r+1's).

    n_local     this rank's number of entries
    density     rho; k = floor(rho N + 1/2) clamped to [0, N], N over all ranks
    local_hist  (prefix, pshift, shift, nbins) -> counts of this rank's keys
                with key >> pshift == prefix, binned by (key >> shift) &
                (nbins - 1); on a GPU, the library's radix histogram of the
                rank's range
    local_ties  t -> number of this rank's keys equal to t

    Collectives: one all-reduce of n (int64), one all-reduce of at most 2048
    int64 counters per radix level (three levels), one all-gather of one
    int64.  Every rank returns the same unit figures."""
    import torch
    import torch.distributed as dist

    def allreduce(x):
        t = torch.as_tensor(x, dtype=torch.int64).clone()
        dist.all_reduce(t, group=group)
        return t

    n_all = int(allreduce([int(n_local)])[0])
    kk = max(0, min(n_all, int(math.floor(density * n_all + 0.5))))
    if kk == 0:
        return SplitSelect(0, 0xFFFFFFFF, 0, 0, 0, 0)
    r = kk                      # rank of the threshold among keys with the current prefix
    prefix, pshift = 0, 31
    last = 0
    for bits in _DIGITS:
        shift = pshift - bits
        nb = 1 << bits
        h = allreduce(list(local_hist(prefix, pshift, shift, nb))).tolist()
        above = 0
        b = nb - 1
        while b > 0 and above + h[b] < r:
            above += h[b]
            b -= 1
        r -= above
        prefix = (prefix << bits) | b
        pshift = shift
        last = h[b]
    t = prefix
    need = r                    # ties at t the unit keeps; k - need keys lie above t
    mine = int(local_ties(t))
    world = dist.get_world_size(group)
    got = [torch.zeros(1, dtype=torch.int64) for _ in range(world)]
    dist.all_gather(got, torch.tensor([mine], dtype=torch.int64), group=group)
    me = dist.get_rank(group)
    before = sum(int(x[0]) for x in got[:me])
    take = max(0, min(mine, need - before))
    return SplitSelect(kk, t, kk - need, int(last), need, take)
