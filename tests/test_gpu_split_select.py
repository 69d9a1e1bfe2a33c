"""The device side of a selection unit split over ranks (App. F, TIES trim
under the global magnitude density): iso_range_hist and iso_range_mask
through the C ABI, against the oracle's binary32 task vector and its
whole-unit TopKMask.

* the radix counts of a range (odd begin and end, every digit level the
  host descent uses, the tie count) equal numpy's counts of the oracle's keys;
* the mask words of every range of a split equal the oracle's whole-unit mask
  restricted to the range, with the unit's ties shared out lowest position
  first;
* two ranks (gloo, one process each, both on this GPU; the kernels never wait
  on one another, only the host exchanges counts) each hold one part of a
  unit with heavy ties, find its threshold through shard.split_unit_select
  with the library's histogram, and write masks that stitch into the
  oracle's mask of the whole unit.
"""
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest
import torch

import oracle
import paper_2607_19331_gb300 as iso

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)


def _bits(t):
    return t.view(torch.int16).numpy().view(np.uint16) if t.dtype == torch.bfloat16 else t.numpy()


def _unit(seed, n, ckpt):
    """A unit with bf16-quantised deltas (long runs of equal keys) and exact
    zeros: (x, base or None) on the host and the oracle's binary32 tau."""
    g = torch.Generator().manual_seed(seed)
    base = (torch.randn(n, generator=g) * 0.02).to(torch.bfloat16)
    d = torch.randn(n, generator=g) * 1e-3
    d[torch.rand(n, generator=g) < 0.05] = 0.0
    if ckpt:
        x = (base.float() + d).to(torch.bfloat16)
        tau32, _ = oracle.delta(_bits(x), _bits(base))
        return x, base, tau32
    x = (torch.round(d * 2 ** 14) / 2 ** 14).float()
    tau32, _ = oracle.delta(_bits(x), np.zeros(n, np.float32))
    return x, None, tau32


def _keys(tau32):
    return tau32.view(np.uint32).astype(np.int64) & 0x7FFFFFFF


def _unpack(words, n):
    w = words.cpu().numpy().view(np.uint32)
    bits = (w[:, None] >> np.arange(32, dtype=np.uint32)) & 1
    return bits.ravel()[:n].astype(np.uint8)


@pytest.mark.parametrize("ckpt", [True, False])
def test_range_hist_matches_oracle_keys(ckpt):
    n = 300_001
    x, base, tau32 = _unit(11, n, ckpt)
    keys = _keys(tau32)
    xd = x.to(DEV)
    bd = base.to(DEV) if base is not None else None
    for b, e in ((0, n), (7, 299_993), (123_457, 123_458), (5, 5)):
        k = keys[b:e]
        # the first level of the host descent, then a deeper digit under a
        # populated prefix, then the last 9 bits
        got = iso.range_hist(xd, bd, b, e, 0, 31, 20, 2048).cpu().numpy()
        assert np.array_equal(got, np.bincount(k >> 20, minlength=2048)[:2048]), (b, e)
        if e > b:
            p1 = int(np.bincount(k >> 20).argmax())
            got = iso.range_hist(xd, bd, b, e, p1, 20, 9, 2048).cpu().numpy()
            sel = k[(k >> 20) == p1]
            assert np.array_equal(got, np.bincount((sel >> 9) & 2047, minlength=2048)), (b, e)
            p2 = int((p1 << 11) | np.bincount((sel >> 9) & 2047).argmax())
            got = iso.range_hist(xd, bd, b, e, p2, 9, 0, 512).cpu().numpy()
            sel = k[(k >> 9) == p2]
            assert np.array_equal(got, np.bincount(sel & 511, minlength=512)), (b, e)
            t = int(k[len(k) // 2])
            got = iso.range_hist(xd, bd, b, e, t, 0, 0, 1).cpu().numpy()
            assert got[0] == int(np.sum(k == t)), (b, e)


@pytest.mark.parametrize("rho", [0.0, 0.05, 0.2, 1.0, 1e-5])
def test_range_masks_stitch_into_the_unit_mask(rho):
    n = 1_000_003
    x, base, tau32 = _unit(12, n, True)
    want, st = oracle.topk_unit(tau32, oracle.k_of(rho, n))
    keys = _keys(tau32)
    t = int(st["thresh_key"])
    need = int(st["ties_taken"])
    xd, bd = x.to(DEV), base.to(DEV)
    bounds = [0, 1, 333_333, 333_365, 900_001, n]
    before = 0
    for b, e in zip(bounds[:-1], bounds[1:]):
        mine = int(np.sum(keys[b:e] == t)) if st["k"] > 0 else 0
        take = max(0, min(mine, need - before))
        before += mine
        got = _unpack(iso.range_mask(xd, t, take, bd, b, e), e - b)
        assert np.array_equal(got, want[b:e]), (rho, b, e)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q, n, bounds, densities):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        torch.cuda.set_device(0)
        x, base, _ = _unit(13, n, True)
        b, e = bounds[rank], bounds[rank + 1]
        # this rank holds only its part of the unit
        xd, bd = x[b:e].contiguous().to(DEV), base[b:e].contiguous().to(DEV)
        out = []
        for rho in densities:
            sel, words = iso.split_unit_topk(xd, rho, bd)
            torch.cuda.synchronize()
            out.append((rho, (sel.k, sel.t, sel.count_above, sel.ties_at_thresh, sel.ties_taken),
                        _unpack(words, e - b)))
        q.put((rank, out))
    finally:
        dist.destroy_process_group()


def test_two_ranks_select_one_unit_through_the_library():
    n = 2_000_017
    bounds = [0, 1_234_567, n]
    densities = [0.05, 0.2, 3e-6]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q, n, bounds, densities)) for r in range(2)]
    for p in procs:
        p.start()
    res = dict(q.get(timeout=300) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    _, _, tau32 = _unit(13, n, True)
    for j, rho in enumerate(densities):
        want, st = oracle.topk_unit(tau32, oracle.k_of(rho, n))
        stitched = np.concatenate([res[r][j][2] for r in range(2)])
        assert np.array_equal(stitched, want), rho
        for r in range(2):
            k, t, above, ties, taken = res[r][j][1]
            assert k == st["k"] and t == st["thresh_key"] and above == st["count_above"]
            assert ties == st["ties_at_thresh"] and taken == st["ties_taken"]
        assert st["ties_at_thresh"] > st["ties_taken"] > 0 or rho < 1e-5    # ties really split
