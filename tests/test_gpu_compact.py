"""K >= 2 TIES and ISO merges through the compact candidates.

The counting pass writes each expert's values at or above the low edge of its
sampled band (with a bit mask per tile), and the Gram and merge passes read
those instead of the full task vectors (iso_compact_candidates; off by
default, since on GB300 the full passes measured faster).  These tests check, through the C ABI, that
* the merged outputs are bit for bit those of the full passes (TIES, and ISO
  with binary32 experts, whose Gram sums run in the same order), and within
  the oracle's tolerances for every case;
* the units report that they took the compact path (unit flag bit 5);
* a unit whose candidates overflow their segment (task vectors on a coarse
  grid: long runs of equal keys at the band's edge) falls back to the full
  task vector for that expert and still matches the oracle.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_19331_gb300 as iso
import synth
from paper_2607_19331_gb300 import _abi
from parity_util import assert_units_equal, assert_values_close, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
SHAPES = synth.qwen_shapes("qwen1.5b", layers=2, scale=4)
OPS = {"ties": oracle.TIES, "iso": oracle.ISO}


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()
    yield
    iso.compact_candidates(False)


def _np(ts):
    return [to_np(t) for t in ts]


def _run(th0, experts, op, density, deltas, compact):
    iso.compact_candidates(compact)
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in experts]
    out, st = iso.iso_merge(d0, dx, op=op, experts_are_deltas=deltas, density=density, stats=True)
    torch.cuda.synchronize()
    return [t.cpu() for t in out], st


def _bits(ts):
    return [t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32) for t in ts]


def _check_oracle(out, st, th0, experts, op, density, deltas, K):
    r = oracle.merge(_np(th0), [_np(e) for e in experts], OPS[op], experts_are_deltas=deltas, density=density,
                     shapes=[(a, b) for a, b, _ in SHAPES], is_1d=[o for _, _, o in SHAPES])
    for q, o in enumerate(out):
        assert_values_close(to_np(o), r["out64"][q], r["mag"][q], f"compact {op} K={K} tensor {q}", op=op, K=K)
    assert int(st.status.item()) == 0
    assert_units_equal(st.units_numpy(), r["units"], f"compact {op} K={K}")


@pytest.mark.parametrize("op", ["ties", "iso"])
@pytest.mark.parametrize("K,inputs", [(2, "f32"), (5, "f32"), (8, "f32"), (3, "ckpt"), (8, "ckpt")])
def test_compact_merge_equals_full_passes(op, K, inputs):
    density = 0.1
    if inputs == "f32":
        th0 = synth.base_weights(SHAPES, seed=61)
        taus, _ = synth.merge_experts(SHAPES, seed=61, K=K)
        experts, deltas = taus, True
    else:
        # each expert an RL checkpoint of the one base, bf16(theta_0 + delta_i),
        # with its own delta
        th0 = synth.base_weights(SHAPES, seed=62)
        experts = []
        for i in range(K):
            row = []
            for q, (sh, w) in enumerate(zip(SHAPES, th0)):
                g = torch.Generator().manual_seed(62_000 + 131 * i + q)
                d = synth.rl_delta(sh, g, "cpu")
                row.append((w.reshape(-1).float() + d).to(torch.bfloat16).reshape(w.shape))
            experts.append(row)
        deltas = False
    out_c, st_c = _run(th0, experts, op, density, deltas, True)
    out_f, st_f = _run(th0, experts, op, density, deltas, False)
    flags = st_c.units_numpy()["flags"]
    ks = st_c.units_numpy()["k"]
    assert ((flags & 32) != 0)[ks > 0].mean() > 0.9, "the compact path was not taken"
    assert not (st_f.units_numpy()["flags"] & 32).any()
    if op == "ties" or inputs == "f32":
        for q, (a, b) in enumerate(zip(_bits(out_c), _bits(out_f))):
            assert torch.equal(a, b), f"{op} K={K} {inputs}: tensor {q} differs from the full passes"
    _check_oracle(out_c, st_c, th0, experts, op, density, deltas, K)


def test_compact_overflow_falls_back_per_expert():
    # task vectors on a coarse grid: few distinct magnitudes, so the band's
    # low edge carries a long run of equal keys and the values at or above it
    # outgrow the segment sized for binary32 task vectors
    K, density = 4, 0.2
    th0 = synth.base_weights(SHAPES, seed=63)
    experts = []
    for i in range(K):
        g = torch.Generator().manual_seed(630 + i)
        row = []
        for r, c, one in SHAPES:
            x = torch.round(torch.randn(r * c, generator=g) * 1e-3 * 600) / 600
            row.append(x.reshape(c) if one else x.reshape(r, c))
        experts.append(row)
    out, st = _run(th0, experts, "ties", density, True, True)
    flags = st.units_numpy()["flags"]
    ks = st.units_numpy()["k"]
    assert ((flags & 32) == 0)[ks > 0].any(), "no unit fell back"
    _check_oracle(out, st, th0, experts, "ties", density, True, K)
