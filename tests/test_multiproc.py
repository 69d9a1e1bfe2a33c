"""The host logic of runs on several GPUs, as world-size-2 gloo process
groups on the CPU: whole-tensor sharding (no data-path collective) and the
step time taken as the maximum over ranks."""
import os
import socket

import pytest
import torch.multiprocessing as mp

from paper_2607_19331_gb300.shard import job_throughput, reduce_step_ms, shard_tensors
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
