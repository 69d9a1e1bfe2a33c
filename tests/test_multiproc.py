"""The host logic of runs on several GPUs, as gloo process groups on the
CPU: whole-tensor sharding (no data-path collective), the step time taken as
the maximum over ranks, and the exchange step of a selection unit split over
ranks (histogram all-reduce per radix level, tie-count all-gather), whose
stitched masks must equal the oracle's TopKMask of the whole unit."""
import os
import socket

import pytest
import torch.multiprocessing as mp

import numpy as np

from paper_2607_19331_gb300.shard import job_throughput, reduce_step_ms, shard_tensors, split_unit_select
import synth


def test_shard_tensors_covers_every_tensor_once_and_balances():
    shapes = synth.qwen_shapes("qwen7b")
    numels = [r * c for r, c, _ in shapes]
    for world in (1, 2, 4, 8):
        parts = shard_tensors(numels, world)
        flat = sorted(q for p in parts for q in p)
        assert flat == list(range(len(numels)))
        loads = [sum(numels[q] for q in p) for p in parts]
        # greedy largest-first: no rank exceeds the mean by more than the largest tensor
        assert max(loads) - sum(loads) / world <= max(numels)
        for p in parts:
            assert p == sorted(p)
    assert shard_tensors([5, 0, 3], 2) == shard_tensors([5, 0, 3], 2)


def test_shard_tensors_rejects_empty_world():
    with pytest.raises(ValueError):
        shard_tensors([1, 2], 0)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        shapes = synth.qwen_shapes("qwen1.5b", layers=2, scale=8)
        numels = [r * c for r, c, _ in shapes]
        mine = shard_tensors(numels, world)[rank]
        ms = 1.0 + rank                       # rank 1 is the slower one
        step = reduce_step_ms(ms)
        n_all = [0]
        import torch
        t = torch.tensor([sum(numels[i] for i in mine)], dtype=torch.int64)
        dist.all_reduce(t)
        n_all = int(t.item())
        q.put((rank, step, n_all, sum(numels), mine))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo_step_time_is_the_maximum():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    assert all(step == 2.0 for _, step, _, _, _ in res)
    assert all(n_all == total for _, _, n_all, total, _ in res)
    assert not set(res[0][4]) & set(res[1][4])
    assert job_throughput(2 * 10**9, 2.0) == pytest.approx(1000.0)
    assert reduce_step_ms(3.5) == 3.5        # no process group in this process


def _unit_keys(seed, n):
    """A task vector with bf16-quantised values (long runs of exact ties) and
    some exact zeros, as binary32; its magnitude keys."""
    rng = np.random.default_rng(seed)
    x = rng.normal(0, 1e-3, n).astype(np.float32)
    x = np.round(x * 2 ** 14) / 2 ** 14            # few distinct magnitudes
    x[rng.random(n) < 0.05] = 0.0
    return x.astype(np.float32), x.astype(np.float32).view(np.uint32) & np.uint32(0x7FFFFFFF)


def _split_worker(rank, world, port, q, seed, n, bounds, densities):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        _, keys = _unit_keys(seed, n)
        mine = keys[bounds[rank]:bounds[rank + 1]].astype(np.int64)

        def local_hist(prefix, pshift, shift, nb):
            sel = mine[(mine >> pshift) == prefix]
            return np.bincount((sel >> shift) & (nb - 1), minlength=nb).tolist()

        def local_ties(t):
            return int(np.sum(mine == t))

        out = []
        for rho in densities:
            s = split_unit_select(mine.size, rho, local_hist, local_ties)
            tie = mine == s.t
            mask = (mine > s.t) | (tie & (np.cumsum(tie) <= s.take))
            out.append((rho, s, mask.astype(np.uint8)))
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world,bounds", [(2, [0, 3000, 7001]), (3, [0, 2500, 2500, 7001]),
                                          (4, [0, 1, 4000, 6999, 7001])])
def test_split_unit_select_matches_whole_unit(world, bounds):
    import oracle
    n, seed = 7001, 5
    densities = [0.0, 0.05, 0.2, 0.5, 1.0, 1.0 / 7001]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_split_worker, args=(r, world, port, q, seed, n, bounds, densities))
             for r in range(world)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=180) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    tau, _ = _unit_keys(seed, n)
    for j, rho in enumerate(densities):
        m_want, st = oracle.topk_unit(tau, oracle.k_of(rho, n))
        stitched = np.concatenate([res[r][j][2] for r in range(world)])
        assert np.array_equal(stitched, m_want), f"rho={rho}"
        for r in range(world):
            s = res[r][j][1]
            assert s.k == st["k"] and s.t == st["thresh_key"]
            assert s.count_above == st["count_above"]
            if s.k:
                assert s.ties_at_thresh == st["ties_at_thresh"] and s.ties_taken == st["ties_taken"]
        if 0.0 < rho < 1.0 and rho * n > 100:
            assert st["ties_at_thresh"] > st["ties_taken"] > 0      # the tie rule really splits ties
