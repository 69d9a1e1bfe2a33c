"""iso_update_host: the K = 1 update of a parameter set in host memory,
pipelined over tensor groups (copies in, update, copies out on three streams).

The call runs the same kernels as iso_update on device copies of each group,
so the tests hold it to identical bits against iso_update on the same inputs
(whose parity with the oracle the other GPU tests establish), with the
device-side statistics of the whole list, for every operator and scope, small
groups that cycle both staging slots many times, tensors laid out back to
back (one copy per run) or apart (one copy per tensor), an empty tensor in the
list, in-place output, pageable host memory and a single stream.
"""
import numpy as np
import pytest
import torch

import paper_2607_19331_gb300 as iso
import synth

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
MINI = synth.qwen_shapes("qwen1.5b", layers=2, scale=8)


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)


def _flat(ts, pin=True):
    """Copies of ts as views of one host buffer, back to back on 16-byte
    boundaries."""
    step = 16 // ts[0].element_size()
    offs, o = [], 0
    for t in ts:
        offs.append(o)
        o += -(-t.numel() // step) * step
    buf = torch.empty(max(1, o), dtype=ts[0].dtype, pin_memory=pin)
    out = [buf[a:a + t.numel()].view(t.shape) for a, t in zip(offs, ts)]
    for v, t in zip(out, ts):
        v.copy_(t)
    return out


def _apart(ts, pin=True):
    return [t.clone().pin_memory() if pin else t.clone() for t in ts]


def _inputs(kind, seed):
    if kind == "ckpt":
        th0, th1 = synth.rl_update_set(MINI, seed=seed)
        return th0, th1, False
    th0 = synth.base_weights(MINI, seed=seed)
    taus, _ = synth.merge_experts(MINI, seed=seed, K=1)
    return th0, taus[0], True


def _device_ref(th0, th1, is_delta, kw):
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    out, st = iso.iso_update(d0, d1, update_is_delta=is_delta, stats=True, **kw)
    torch.cuda.synchronize()
    return [t.cpu() for t in out], st


def _same(a, b, what):
    assert len(a) == len(b)
    for q, (x, y) in enumerate(zip(a, b)):
        assert x.dtype == y.dtype and x.shape == y.shape, (what, q)
        ints = torch.int16 if x.dtype == torch.bfloat16 else torch.int32
        assert torch.equal(x.view(ints), y.view(ints)), f"{what}: tensor {q}"


def _same_stats(st, ref, what):
    assert int(st.status.item()) == 0, what
    a, b = st.units_numpy(), ref.units_numpy()
    # every field of every unit but the diagnostic flags, which record the
    # path the selection took (the fused pass's band records are sized per
    # group of tensors, so a group may take another path to the same result)
    for f in ("thresh_key", "k", "count_above", "ties_at_thresh", "ties_taken"):
        assert np.array_equal(a[f], b[f]), (what, f)
    assert torch.equal(st.gram, ref.gram), what
    assert torch.equal(st.coef, ref.coef), what


@pytest.mark.parametrize("op,scope,kind", [
    ("iso", "tensor", "ckpt"), ("ties", "tensor", "delta"), ("iso", "block", "ckpt"),
    ("ties", "global", "ckpt"), ("ta", "tensor", "delta"), ("ram", "tensor", "ckpt"),
])
@pytest.mark.parametrize("layout", ["flat", "apart"])
def test_host_update_matches_device_update(op, scope, kind, layout):
    th0, th1, is_delta = _inputs(kind, seed=31)
    kw = dict(op=op, scope=scope, density=0.05 if op == "iso" else 0.2)
    ref, st_ref = _device_ref(th0, th1, is_delta, kw)
    mk = _flat if layout == "flat" else _apart
    h0, h1 = mk(th0), mk(th1)
    ho = mk([torch.full_like(t, float("nan")) for t in th0])
    # groups of about 96 KB: the list passes through both slots many times
    host = iso.HostUpdate(DEV, group_bytes=96 << 10)
    out, st = host.run(h0, h1, out=ho, update_is_delta=is_delta, stats=True, **kw)
    torch.cuda.synchronize()
    what = f"host {op} {scope} {kind} {layout}"
    _same(out, ref, what)
    _same_stats(st, st_ref, what)
    assert host.h2d_bytes == sum(t.numel() * t.element_size() for t in th0 + th1)


def test_host_update_in_place_empty_tensor_and_two_calls():
    th0, th1, _ = _inputs("ckpt", seed=32)
    # an empty tensor in the middle of the list takes no copy and no unit work
    cut = len(th0) // 2
    th0 = th0[:cut] + [torch.empty(0, 64, dtype=torch.bfloat16)] + th0[cut:]
    th1 = th1[:cut] + [torch.empty(0, 64, dtype=torch.bfloat16)] + th1[cut:]
    kw = dict(op="iso", density=0.05)
    ref, st_ref = _device_ref(th0, th1, False, kw)
    host = iso.HostUpdate(DEV, group_bytes=200 << 10)
    h0, h1 = _flat(th0), _flat(th1)
    out, st = host.run(h0, h1, out=h0, stats=True, **kw)        # in place over the host base
    torch.cuda.synchronize()
    assert out is h0
    _same(h0, ref, "in place")
    _same_stats(st, st_ref, "in place")
    # a second call with other inputs through the same staging buffer
    g0, g1, _ = _inputs("ckpt", seed=33)
    ref2, _ = _device_ref(g0, g1, False, kw)
    out2 = host.run(_flat(g0), _flat(g1), **kw)
    torch.cuda.synchronize()
    _same(out2, ref2, "second call")


def test_host_update_pageable_memory_and_one_stream():
    th0, th1, is_delta = _inputs("delta", seed=34)
    kw = dict(op="ties", density=0.2)
    ref, _ = _device_ref(th0, th1, is_delta, kw)
    host = iso.HostUpdate(DEV, group_bytes=128 << 10)
    s = torch.cuda.current_stream()
    host.streams = [s, s, s]                 # no overlap: copies and update in order on one stream
    out = host.run(_apart(th0, pin=False), _apart(th1, pin=False), update_is_delta=is_delta,
                   **kw)
    torch.cuda.synchronize()
    _same(out, ref, "pageable, one stream")


def test_host_update_reports_nonfinite_from_a_later_group():
    th0, th1, _ = _inputs("ckpt", seed=35)
    th1[-3] = th1[-3].clone()
    th1[-3].view(-1)[7] = float("inf")
    host = iso.HostUpdate(DEV, group_bytes=64 << 10)
    _, st = host.run(_flat(th0), _flat(th1), op="iso", density=0.05, stats=True)
    torch.cuda.synchronize()
    from paper_2607_19331_gb300 import _abi
    assert int(st.status.item()) == _abi.ISO_ERR_NONFINITE


@pytest.mark.parametrize("op,scope", [("iso", "tensor"), ("iso", "block"), ("ties", "global")])
def test_update_of_untrimmed_tensors_only_writes_their_unit_records(op, scope):
    # a list with no trimmed tensor (ISO leaves 1-D tensors untrimmed; TIES
    # with mask_1d off too) runs no selection pass: its units still get the
    # record of an untrimmed unit
    vecs = [torch.randn(n, device=DEV).to(torch.bfloat16) for n in (96, 1000, 8)]
    upd = [(v.float() + 1e-3).to(torch.bfloat16) for v in vecs]
    _, st = iso.iso_update(vecs, upd, op=op, scope=scope, density=0.2, mask_1d=False, stats=True)
    torch.cuda.synchronize()
    u = st.units_numpy()
    assert u.shape[1] == st.n_units and st.n_units >= 1
    assert (u["thresh_key"] == 0xFFFFFFFF).all() and (u["k"] == -1).all()
    assert (u["count_above"] == 0).all() and (u["ties_taken"] == 0).all()
