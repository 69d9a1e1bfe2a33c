"""iso_update_noalloc: the update for callers that cannot allocate device memory.

Such callers (an inference-engine plugin whose enqueue path may not call
cudaMalloc, a server that freezes its allocator after warm-up, a C host with
no device allocator) cannot pass a workspace; the library then uses its own
fixed per-device scratch.  These tests call that entry point through the C ABI
and check it against iso_update, which takes a caller workspace, on two calls
in a row with different inputs, so a stale value left in the shared scratch by
the first call would show in the second.  The file sorts last so that a run
stopping at the first failure has already run every other test.
"""
import ctypes

import pytest
import torch

import paper_2607_19331_gb300 as iso
import synth
from paper_2607_19331_gb300 import _abi
from paper_2607_19331_gb300.api import describe, make_stats, merge_cfg

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
SHAPES = synth.qwen_shapes("qwen1.5b", layers=2, scale=8)


def _noalloc(th0, th1, cfg, out, st):
    return _abi.lib().iso_update_noalloc(describe(th0), describe(th1), 0, describe(out), len(th0),
                                         ctypes.byref(cfg), ctypes.byref(st.abi()),
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def test_noalloc_matches_workspace_update_on_two_calls():
    assert torch.cuda.is_available()
    from paper_2607_19331_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    for seed, op, density in ((21, "iso", 0.05), (22, "ties", 0.2)):
        th0, th1 = synth.rl_update_set(SHAPES, seed=seed, device=DEV)
        ref, st_ref = iso.iso_update(th0, th1, op=op, density=density, stats=True,
                                     workspace=iso.Workspace(DEV))
        cfg = merge_cfg(op, density)
        out = [torch.full_like(t, float("nan")) for t in th0]
        st = make_stats(th0, 1, cfg.topk, DEV)
        assert _noalloc(th0, th1, cfg, out, st) == _abi.ISO_OK
        torch.cuda.synchronize()
        assert int(st.status.item()) == 0
        for q, (a, b) in enumerate(zip(out, ref)):
            # the same kernels on the same inputs: identical bits, so a value
            # left in the shared scratch by the first call cannot hide
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), f"noalloc {op} tensor {q}"
        assert torch.equal(st.units, st_ref.units)
        assert torch.equal(st.coef, st_ref.coef)


def test_noalloc_rejects_requests_beyond_the_scratch():
    cfg = merge_cfg("iso", 0.05)
    # descriptors only (nothing is launched): three disjoint 800 MB ranges
    big = (_abi.IsoTensor * 1)(_abi.IsoTensor(1 << 40, 20000, 20000, _abi.ISO_BF16, 0))
    upd = (_abi.IsoTensor * 1)(_abi.IsoTensor(2 << 40, 20000, 20000, _abi.ISO_BF16, 0))
    out = (_abi.IsoTensor * 1)(_abi.IsoTensor(3 << 40, 20000, 20000, _abi.ISO_BF16, 0))
    rc = _abi.lib().iso_update_noalloc(big, upd, 0, out, 1, ctypes.byref(cfg), None, None)
    assert rc == _abi.ISO_ERR_WORKSPACE
