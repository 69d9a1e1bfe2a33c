"""GPU parity of the RAM merge (App. F: active set |tau_i| > eps_act, unique
values kept whole, shared ones averaged over the active experts) against the
CPU oracle, through the C ABI.

Activity is decided on the binary32 task vector on both sides, so every
decision agrees exactly; values are compared within the tolerances of
parity_util.  Inputs are seeded and synthetic: bf16 RL checkpoints (whose
bf16-quantised deltas are exactly zero wherever the update is below half an
ulp of the base weight, the sparsity RAM is built for), fp32 task vectors with
a threshold that leaves a third of the entries inactive, and task vectors on a
grid with many entries exactly at the threshold.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_19331_gb300 as iso
import synth
from paper_2607_19331_gb300 import _abi
from parity_util import assert_values_close, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
EPS = float(np.float32(1e-5))   # the paper's eps_act, as the binary32 value the library takes


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()


def _np(ts):
    return [to_np(t) for t in ts]


def _check(out, st, r, theta0, what, K=8):
    torch.cuda.synchronize()
    if st is not None:
        assert int(st.status.item()) == 0, what
    for q, (o, b) in enumerate(zip(out, theta0)):
        g = to_np(o)
        assert g.dtype == (np.uint16 if b.dtype == torch.bfloat16 else np.float32)
        assert_values_close(g, r["out64"][q], r["mag"][q], f"{what} tensor {q}", op="ram", K=K)


MINI = synth.qwen_shapes("qwen1.5b", layers=2, scale=8)
# several tiles and ragged tails, 1-D, tiny and empty tensors
MIXED = [(300, 1000, False), (257, 129, False), (1, 1536, True), (3, 7, False),
         (0, 5, False), (64, 4096, False), (1, 5, True)]


def _shapes(sh):
    return [(r, c) for r, c, _ in sh]


def _is1d(sh):
    return [o for _, _, o in sh]


@pytest.mark.parametrize("K", [2, 3, 4, 5, 8])
@pytest.mark.parametrize("lam", [1.0, 0.6])
def test_ram_merge_bf16_checkpoints(K, lam):
    shapes = synth.qwen_shapes("qwen1.5b", layers=1, scale=8)
    th0 = synth.base_weights(shapes, seed=11)
    cks = []
    for i in range(K):
        # expert i's RL checkpoint over the one base: bf16(theta_0 + delta_i)
        row = []
        for q, (s, w) in enumerate(zip(shapes, th0)):
            g = torch.Generator().manual_seed(20_000 + 131 * i + q)
            d = synth.rl_delta(s, g, "cpu")
            row.append((w.reshape(-1).float() + d).to(torch.bfloat16).reshape(w.shape))
        cks.append(row)
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in cks]
    out, st = iso.iso_merge(d0, dx, op="ram", experts_are_deltas=False, lam=lam, eps_act=EPS,
                            stats=True)
    r = oracle.merge(_np(th0), [_np(e) for e in cks], oracle.RAM, experts_are_deltas=False,
                     lam=lam, eps_act=EPS, shapes=_shapes(shapes), is_1d=_is1d(shapes))
    _check(out, st, r, th0, f"RAM K={K} checkpoints", K=K)
    # the quantised deltas really are sparse: some entries have no active expert
    t = (cks[0][1].float() - th0[1].float()).abs()
    assert 0.0 < float((t <= EPS).float().mean()) < 0.9


@pytest.mark.parametrize("K", [1, 2, 4, 7, 8])
@pytest.mark.parametrize("base_dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("x_dtype", [torch.float32, torch.bfloat16])
def test_ram_merge_task_vectors(K, base_dtype, x_dtype):
    th0 = synth.base_weights(MIXED, seed=3, dtype=base_dtype)
    taus = []
    for i in range(K):
        row = []
        for q, (rr, cc, one) in enumerate(MIXED):
            g = torch.Generator().manual_seed(1000 * i + q)
            x = torch.randn(rr * cc, generator=g) * 5e-4
            x = x.reshape(cc) if one else x.reshape(rr, cc)
            row.append(x.to(x_dtype))
        taus.append(row)
    eps = float(np.float32(2e-4))   # about a third of the entries inactive per expert
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in taus]
    if K == 1:
        out, st = iso.iso_update(d0, dx[0], op="ram", update_is_delta=True, eps_act=eps, stats=True)
    else:
        out, st = iso.iso_merge(d0, dx, op="ram", eps_act=eps, stats=True)
    r = oracle.merge(_np(th0), [_np(e) for e in taus], oracle.RAM, eps_act=eps,
                     shapes=_shapes(MIXED), is_1d=_is1d(MIXED))
    _check(out, st, r, th0, f"RAM K={K} {base_dtype} {x_dtype}", K=K)


@pytest.mark.parametrize("K", [3, 8])
def test_ram_threshold_ties_exact(K):
    # task vectors on a grid of 2^-12 with eps_act = 2^-10 on the grid: many
    # entries sit exactly at the threshold and must count as inactive
    shapes = [(256, 1000, False), (1, 777, True)]
    th0 = synth.base_weights(shapes, seed=5, dtype=torch.float32)
    taus = []
    for i in range(K):
        row = []
        for q, (rr, cc, one) in enumerate(shapes):
            g = torch.Generator().manual_seed(77 * i + q)
            x = torch.randint(-8, 9, (rr * cc,), generator=g).float() * 2.0 ** -12
            row.append(x.reshape(cc) if one else x.reshape(rr, cc))
        taus.append(row)
    eps = 2.0 ** -10
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in taus]
    out, st = iso.iso_merge(d0, dx, op="ram", eps_act=eps, stats=True)
    r = oracle.merge(_np(th0), [_np(e) for e in taus], oracle.RAM, eps_act=eps,
                     shapes=_shapes(shapes), is_1d=_is1d(shapes))
    _check(out, st, r, th0, f"RAM ties K={K}", K=K)
    # dyadic inputs and power-of-two-free counts aside, every kept or dropped
    # decision shows: entries with no active expert are theta_0 bit for bit
    for q in range(len(shapes)):
        act = np.zeros(taus[0][q].numel(), np.int64)
        for i in range(K):
            act += (np.abs(to_np(taus[i][q])) > eps)
        none = act == 0
        assert none.any()
        assert np.array_equal(to_np(out[q])[none], to_np(th0[q])[none])


def test_ram_zero_delta_and_threshold_fixed_point():
    th0 = synth.base_weights(MINI[:4], seed=9)
    th0[0].view(-1)[7] = -0.0
    zeros = [torch.zeros(t.shape, dtype=torch.float32) for t in th0]
    d0 = [t.to(DEV) for t in th0]
    out = iso.iso_merge(d0, [[z.to(DEV) for z in zeros]] * 3, op="ram", eps_act=0.0)
    torch.cuda.synchronize()
    for a, b in zip(out, th0):
        assert torch.equal(a.cpu().view(torch.int16), b.view(torch.int16))
    taus = [[torch.randn(t.shape) * 1e-3 for t in th0] for _ in range(2)]
    big = max(float(x.abs().max()) for e in taus for x in e)
    out = iso.iso_merge(d0, [[x.to(DEV) for x in e] for e in taus], op="ram", eps_act=big)
    torch.cuda.synchronize()
    for a, b in zip(out, th0):
        assert torch.equal(a.cpu().view(torch.int16), b.view(torch.int16))


def test_ram_in_place():
    th0, th1 = synth.rl_update_set(MINI, seed=4)
    d0 = [t.to(DEV) for t in th0]
    ref = iso.iso_update(d0, [t.to(DEV) for t in th1], op="ram", eps_act=EPS)
    got = iso.iso_update(d0, [t.to(DEV) for t in th1], op="ram", eps_act=EPS, out=d0)
    torch.cuda.synchronize()
    for a, b in zip(ref, got):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))


def test_ram_nonfinite_reported():
    th0 = synth.base_weights(MINI[:3], seed=7, dtype=torch.float32)
    taus = [[torch.randn(t.shape) * 1e-3 for t in th0] for _ in range(3)]
    taus[2][1].view(-1)[99] = float("inf")
    _, st = iso.iso_merge([t.to(DEV) for t in th0], [[x.to(DEV) for x in e] for e in taus],
                          op="ram", eps_act=EPS, stats=True)
    torch.cuda.synchronize()
    assert int(st.status.item()) == _abi.ISO_ERR_NONFINITE
