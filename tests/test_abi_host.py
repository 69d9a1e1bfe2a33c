"""Host-side checks of the C ABI (no GPU needed): the library loads, exports
every entry point include/iso.h declares, and rejects bad arguments before
anything reaches the device."""
import ctypes
import os
import re

import pytest

import paper_2607_19331_gb300 as iso
from paper_2607_19331_gb300 import _abi
from paper_2607_19331_gb300._abi import IsoTensor

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2607_19331_gb300 import build
    build.build()


def _declared():
    src = open(os.path.join(ROOT, "include", "iso.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(iso_[a-z_0-9]+)\s*\(", src)))


def test_every_declared_symbol_is_exported():
    names = _declared()
    assert {"iso_delta", "iso_topk_mask", "iso_update", "iso_merge", "iso_workspace_size"} <= set(names)
    lib = ctypes.CDLL(_abi.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), f"{n} declared in iso.h but not exported"
    assert {p[0] for p in _abi.PROTOTYPES} == set(names)


def test_error_strings():
    L = _abi.lib()
    for code in range(0, -10, -1):
        s = L.iso_error_string(code).decode()
        assert s.startswith("ISO_"), s
    assert "unknown" in L.iso_error_string(-99).decode()


def _fake(rows, cols, dtype=_abi.ISO_BF16, ptr=0x10000, is_1d=0):
    return IsoTensor(ptr, rows, cols, dtype, is_1d)


def _arr(*ts):
    a = (IsoTensor * len(ts))()
    for i, t in enumerate(ts):
        a[i] = t
    return a


def test_num_units_and_workspace():
    L = _abi.lib()
    ts = _arr(_fake(300, 1000), _fake(1, 1536, is_1d=1), _fake(257, 129))
    n = ctypes.c_int64()
    for scope, want in ((0, 3), (2, 1), (1, 3 * 8 + 12 + 3 * 2)):
        cfg = iso.topk_cfg(0.1, ["tensor", "block", "global"][scope])
        assert L.iso_num_units(ts, 3, ctypes.byref(cfg), ctypes.byref(n)) == 0
        assert n.value == want, (scope, n.value)
    mn, full = ctypes.c_size_t(), ctypes.c_size_t()
    for op in ("ta", "ties", "iso", "ram"):
        for scope in ("tensor", "block", "global"):
            cfg = iso.merge_cfg(op, 0.05, scope)
            assert L.iso_workspace_size(ts, 3, 2, ctypes.byref(cfg), ctypes.byref(mn), ctypes.byref(full)) == 0
            assert 0 < mn.value <= full.value
            if scope == "global" and op not in ("ta", "ram"):
                assert mn.value == full.value
    cfg = iso.merge_cfg("ties", 0.05)
    assert L.iso_workspace_size(ts, 3, 9, ctypes.byref(cfg), None, None) == _abi.ISO_ERR_UNSUPPORTED


def test_validation_rejects_before_launch():
    L = _abi.lib()
    cfg = iso.merge_cfg("ties", 0.2)
    a, b = _arr(_fake(8, 8)), _arr(_fake(8, 8, ptr=0x20000))
    o = _arr(_fake(8, 8, ptr=0x30000))
    ws = ctypes.c_void_p(0x40000)
    def upd(a_, b_, o_, cfg_=cfg, ws_=ws, n=1):
        return L.iso_update(a_, b_, 0, o_, n, ctypes.byref(cfg_) if cfg_ is not None else None,
                            ws_, 1 << 20, None, None)
    assert upd(a, _arr(_fake(8, 4, ptr=0x20000)), o) == _abi.ISO_ERR_SHAPE
    assert upd(a, _arr(_fake(8, 8, ptr=0x20002)), o) == _abi.ISO_ERR_ALIGN
    assert upd(a, _arr(_fake(8, 8, dtype=7, ptr=0x20000)), o) == _abi.ISO_ERR_DTYPE
    assert upd(a, b, _arr(_fake(8, 8, dtype=_abi.ISO_F32, ptr=0x30000))) == _abi.ISO_ERR_DTYPE
    assert upd(a, b, _arr(_fake(8, 8, ptr=0x20000))) == _abi.ISO_ERR_ARG        # out aliases expert
    assert upd(a, b, o, cfg_=None) == _abi.ISO_ERR_ARG
    assert upd(a, _arr(_fake(8, 8, ptr=0)), o) == _abi.ISO_ERR_ARG               # NULL data
    assert upd(a, b, o, ws_=ctypes.c_void_p(0x40010)) == _abi.ISO_ERR_WORKSPACE  # misaligned
    assert upd(a, b, o, ws_=ctypes.c_void_p(0)) == _abi.ISO_ERR_WORKSPACE
    bad = iso.merge_cfg("ties", 0.2)
    bad.topk.density = float("nan")
    assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_ARG
    bad = iso.merge_cfg("iso", 0.2, c_min=2.0, c_max=1.0)
    assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_ARG
    for eps in (-1e-5, float("nan"), float("inf")):       # RAM threshold: finite, >= 0
        bad = iso.merge_cfg("ram", eps_act=eps)
        assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_ARG
    bad = iso.merge_cfg("ties", 0.2)
    bad.op = 4
    assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_ARG
    # RAM ignores the TopKMask settings (host-only sizing call)
    ram = iso.merge_cfg("ram", 0.2, "block", block=(128, 12))
    assert L.iso_workspace_size(a, 1, 2, ctypes.byref(ram), None, None) == 0
    bad = iso.merge_cfg("ties", 0.2, "block", block=(128, 12))
    assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_ARG
    bad = iso.merge_cfg("ties", 0.2, "block", block=(256, 256))
    assert upd(a, b, o, cfg_=bad) == _abi.ISO_ERR_UNSUPPORTED
    huge = _arr(_fake(1 << 16, 1 << 16))
    assert upd(huge, _arr(_fake(1 << 16, 1 << 16, ptr=0x20000)), _arr(_fake(1 << 16, 1 << 16, ptr=0x30000))) \
        == _abi.ISO_ERR_UNSUPPORTED
    # extents whose product wraps 64 bits (2^33 x 2^31 = 2^64 -> 0) are rejected
    # before the product is formed
    wrap = _arr(_fake(1 << 33, 1 << 31))
    assert upd(wrap, _arr(_fake(1 << 33, 1 << 31, ptr=0x20000)), _arr(_fake(1 << 33, 1 << 31, ptr=0x30000))) \
        == _abi.ISO_ERR_UNSUPPORTED
    assert upd(_arr(_fake(1, 1 << 32)), _arr(_fake(1, 1 << 32, ptr=0x20000)),
               _arr(_fake(1, 1 << 32, ptr=0x30000))) == _abi.ISO_ERR_UNSUPPORTED
    # out may coincide with its own base (in place; tested on the GPU), and overlap nothing else
    assert upd(a, b, _arr(_fake(8, 8, ptr=0x10010))) == _abi.ISO_ERR_ARG            # partial overlap with the base
    assert upd(a, b, _arr(_fake(8, 8, ptr=0x20000 + 64))) == _abi.ISO_ERR_ARG       # partial overlap with the expert
    two_b = _arr(_fake(8, 8), _fake(8, 8, ptr=0x11000))
    two_x = _arr(_fake(8, 8, ptr=0x20000), _fake(8, 8, ptr=0x21000))
    assert upd(two_b, two_x, _arr(_fake(8, 8, ptr=0x30000), _fake(8, 8, ptr=0x20000 + 96)), n=2) \
        == _abi.ISO_ERR_ARG                                                          # out[1] inside expert 0
    assert upd(two_b, two_x, _arr(_fake(8, 8, ptr=0x30000), _fake(8, 8, ptr=0x10000)), n=2) \
        == _abi.ISO_ERR_ARG                                                          # out[1] on base[0]
    assert upd(two_b, two_x, _arr(_fake(8, 8, ptr=0x30000), _fake(8, 8, ptr=0x30040)), n=2) \
        == _abi.ISO_ERR_ARG                                                          # outputs overlap
    K9 = (IsoTensor * 9)(*[_fake(8, 8, ptr=0x50000 + 0x1000 * i) for i in range(9)])
    assert L.iso_merge(a, K9, 9, 1, o, 1, ctypes.byref(cfg), ws, 1 << 20, None, None) == _abi.ISO_ERR_UNSUPPORTED
    # an empty list is a no-op that needs no workspace and no device
    assert L.iso_update(a, b, 0, o, 0, ctypes.byref(cfg), None, 0, None, None) == 0


def test_missing_library_fails_loudly(monkeypatch):
    monkeypatch.setattr(_abi, "LIB_PATH", "/nonexistent/libiso_gb300.so")
    monkeypatch.setattr(_abi, "_lib", None)
    with pytest.raises(RuntimeError, match="not found"):
        _abi.lib()


C_CLIENT = r"""
#include "iso.h"
#include <stdio.h>
int main(void) {
    iso_tensor t = {0};
    t.data = (void*)0x10000; t.rows = 300; t.cols = 1000; t.dtype = ISO_BF16; t.is_1d = 0;
    iso_merge_cfg c = {0};
    c.op = ISO_OP_RAM; c.lambda = 1.0f; c.eps_act = 1e-5f; c.ridge = 1e-12; c.c_min = 0.0; c.c_max = 1.5;
    c.topk.density = 0.2; c.topk.scope = ISO_SCOPE_BLOCK; c.topk.block_rows = 128; c.topk.block_cols = 128;
    size_t mn = 0, full = 0;
    int rc = iso_workspace_size(&t, 1, 2, &c, &mn, &full);
    int64_t nu = 0;
    int rc2 = iso_num_units(&t, 1, &c.topk, &nu);
    c.eps_act = -1.0f;
    int rc3 = iso_workspace_size(&t, 1, 2, &c, &mn, &full);
    printf("%d %d %lld %d\n", rc, rc2, (long long)nu, rc3);
    return (rc == ISO_OK && rc2 == ISO_OK && nu == 3 * 8 && rc3 == ISO_ERR_ARG && full >= mn && mn > 0) ? 0 : 1;
}
"""


def test_header_is_plain_c(tmp_path):
    """include/iso.h compiles as strict C99 and a C program links against the
    library and calls its host-only entry points (no device work)."""
    import shutil
    import subprocess
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not available")
    src = tmp_path / "client.c"
    src.write_text(C_CLIENT)
    exe = tmp_path / "client"
    libdir = os.path.dirname(_abi.LIB_PATH)
    subprocess.check_call([gcc, "-std=c99", "-Wall", "-Wextra", "-pedantic", "-Werror",
                           "-I", os.path.join(ROOT, "include"), "-o", str(exe), str(src),
                           "-L", libdir, "-liso_gb300", f"-Wl,-rpath,{libdir}"])
    r = subprocess.run([str(exe)], capture_output=True, text=True, timeout=60)
    assert r.returncode == 0, r.stdout + r.stderr


def test_workspace_at_full_model_sizes():
    """Host-only sizing at the Qwen2.5-7B shapes (254 tensors, 7.6e9 entries):
    one GLOBAL unit over the whole task vector plans as one group of a few
    GB; per-tensor scopes can run in groups down to the largest tensor; RAM,
    which selects nothing, needs only the tables; a tensor of 2^32 entries is
    refused."""
    import synth
    L = _abi.lib()
    shapes = synth.qwen_shapes("qwen7b")
    mn, full = ctypes.c_size_t(), ctypes.c_size_t()

    def size(op, scope, K, dtype, density):
        ts = _arr(*[_fake(r, c, dtype=dtype, is_1d=int(o)) for r, c, o in shapes])
        cfg = iso.merge_cfg(op, density, scope)
        rc = L.iso_workspace_size(ts, len(shapes), K, ctypes.byref(cfg), ctypes.byref(mn), ctypes.byref(full))
        assert rc == 0, (op, scope, rc)
        return mn.value, full.value

    g_mn, g_full = size("ties", "global", 1, _abi.ISO_BF16, 0.2)
    assert g_mn == g_full and 1e9 < g_full < 8e9
    t_mn, t_full = size("iso", "tensor", 1, _abi.ISO_BF16, 0.05)
    assert t_mn < t_full < 20e9
    # eight experts: the full passes (the default) need a few GB per group;
    # with compact candidates the full size also holds every expert's
    # candidate values (about 15 % of its entries as binary32 plus a bit per
    # entry), while the smallest workspace stays that of the full passes
    k_mn, k_full = size("ties", "tensor", 8, _abi.ISO_F32, 0.1)
    assert k_mn < k_full < 20e9
    iso.compact_candidates(True)
    try:
        k_mn2, k_full2 = size("ties", "tensor", 8, _abi.ISO_F32, 0.1)
    finally:
        iso.compact_candidates(False)
    assert k_mn2 == k_mn and k_full2 < 80e9 and k_full2 - k_full > 30e9
    r_mn, r_full = size("ram", "tensor", 8, _abi.ISO_F32, 0.0)
    assert r_full < (1 << 20)
    cfg = iso.merge_cfg("ties", 0.1)
    big = _arr(_fake(1 << 16, 1 << 16))
    assert L.iso_workspace_size(big, 1, 1, ctypes.byref(cfg), None, None) == _abi.ISO_ERR_UNSUPPORTED


def test_frame_merge_sizes_and_argument_errors():
    # iso_frame_merge: sizing and the checks made before anything is enqueued
    # (descriptors and fake device pointers only; nothing is launched)
    L = _abi.lib()
    b = ctypes.c_size_t()
    assert L.iso_frame_workspace_size(3584, 18944, 8, ctypes.byref(b)) == 0
    assert 10e9 < b.value < 40e9           # the 7B gate/up projection fits the device several times
    small = ctypes.c_size_t()
    assert L.iso_frame_workspace_size(96, 64, 3, ctypes.byref(small)) == 0
    assert 0 < small.value < b.value
    assert L.iso_frame_workspace_size(96, 64, 9, ctypes.byref(small)) == _abi.ISO_ERR_UNSUPPORTED
    assert L.iso_frame_workspace_size(0, 64, 1, ctypes.byref(small)) == _abi.ISO_ERR_ARG
    cfg = _abi.IsoFrameCfg(0.9, 1e-12, 0.0, 1.5, 0, 0)
    P = ctypes.c_void_p
    U = (P * 2)(0x100000, 0x200000)
    V = (P * 2)(0x300000, 0x400000)
    W = _arr(_fake(96, 64, dtype=_abi.ISO_F32, ptr=0x1000000))
    O = _arr(_fake(96, 64, dtype=_abi.ISO_F32, ptr=0x2000000))
    ws = P(0x4000000)

    def fm(W_=W, O_=O, cfg_=cfg, ws_=ws, wsb=1 << 30, m=96, n=64, K=2, U_=U):
        return L.iso_frame_merge(P(0x10000), P(0x20000), P(0x30000), U_, V, K, m, n, W_, O_,
                                 ctypes.byref(cfg_) if cfg_ is not None else None, ws_, wsb, None, None)
    assert fm(W_=_arr(_fake(96, 65, dtype=_abi.ISO_F32, ptr=0x1000000))) == _abi.ISO_ERR_SHAPE
    assert fm(O_=_arr(_fake(96, 64, dtype=_abi.ISO_BF16, ptr=0x2000000))) == _abi.ISO_ERR_DTYPE
    assert fm(O_=_arr(_fake(96, 64, dtype=_abi.ISO_F32, ptr=0x1000040))) == _abi.ISO_ERR_ARG   # overlaps W0
    assert fm(cfg_=None) == _abi.ISO_ERR_ARG
    assert fm(cfg_=_abi.IsoFrameCfg(0.0, 1e-12, 0.0, 1.5, 0, 0)) == _abi.ISO_ERR_ARG           # rho_keep
    assert fm(cfg_=_abi.IsoFrameCfg(0.9, 1e-12, 2.0, 1.5, 0, 0)) == _abi.ISO_ERR_ARG           # clip range
    assert fm(cfg_=_abi.IsoFrameCfg(0.9, 1e-12, 0.0, 1.5, 65, 0)) == _abi.ISO_ERR_ARG          # iterations
    assert fm(ws_=P(0x4000010)) == _abi.ISO_ERR_WORKSPACE                                       # misaligned
    assert fm(wsb=1024) == _abi.ISO_ERR_WORKSPACE
    assert fm(U_=(P * 2)(0x100000, 0)) == _abi.ISO_ERR_ARG
    assert fm(U_=(P * 2)(0x100000, 0x200004)) == _abi.ISO_ERR_ALIGN
    assert fm(K=9) == _abi.ISO_ERR_UNSUPPORTED


def test_gemm_argument_errors():
    L = _abi.lib()
    P = ctypes.c_void_p
    A, B, C = P(0x100000), P(0x200000), P(0x300000)
    assert L.iso_gemm_tf32(A, 32, B, 32, C, 128, 100, 128, 32, 0, 0, None) == _abi.ISO_ERR_SHAPE   # M
    assert L.iso_gemm_tf32(A, 32, B, 32, C, 128, 128, 128, 40, 0, 0, None) == _abi.ISO_ERR_SHAPE   # Kc
    assert L.iso_gemm_tf32(A, 32, B, 32, C, 128, 128, 128, 32, 32, 0, None) == _abi.ISO_ERR_SHAPE  # past lda
    assert L.iso_gemm_tf32(P(0x100004), 32, B, 32, C, 128, 128, 128, 32, 0, 0, None) == _abi.ISO_ERR_ALIGN
    assert L.iso_gemm_tf32(None, 32, B, 32, C, 128, 128, 128, 32, 0, 0, None) == _abi.ISO_ERR_ARG


def test_opt_step_sizes_and_argument_errors():
    # iso_opt_step: sizing and the checks made before anything is enqueued
    L = _abi.lib()
    b = ctypes.c_size_t()
    assert L.iso_opt_workspace_size(3584, 18944, ctypes.byref(b)) == 0
    assert 5e9 < b.value < 40e9
    assert L.iso_opt_workspace_size(0, 5, ctypes.byref(b)) == _abi.ISO_ERR_ARG
    P = ctypes.c_void_p
    G = _arr(_fake(96, 64, dtype=_abi.ISO_F32, ptr=0x1000000))
    W = _arr(_fake(96, 64, dtype=_abi.ISO_BF16, ptr=0x2000000))
    O = _arr(_fake(96, 64, dtype=_abi.ISO_BF16, ptr=0x3000000))

    def cfg(**kw):
        d = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, step=1, ns_iters=0, reserved=0)
        d.update(kw)
        return _abi.IsoAdamwCfg(**d)

    def st(c=None, G_=G, W_=W, O_=O, wsb=1 << 30, U=0x100000, mU=0x500000):
        c = cfg() if c is None else c
        return L.iso_opt_step(P(U), P(0x200000), P(0x300000), G_, P(mU), P(0x600000), P(0x700000),
                              P(0x800000), W_, O_, 96, 64, ctypes.byref(c), P(0x4000000), wsb, None, None)
    assert st(G_=_arr(_fake(96, 65, dtype=_abi.ISO_F32, ptr=0x1000000))) == _abi.ISO_ERR_SHAPE
    assert st(O_=_arr(_fake(96, 64, dtype=_abi.ISO_F32, ptr=0x3000000))) == _abi.ISO_ERR_DTYPE
    assert st(O_=_arr(_fake(96, 64, dtype=_abi.ISO_BF16, ptr=0x2000010))) == _abi.ISO_ERR_ARG     # overlaps W
    assert st(cfg(step=0)) == _abi.ISO_ERR_ARG
    assert st(cfg(beta1=1.0)) == _abi.ISO_ERR_ARG
    assert st(cfg(eps=0.0)) == _abi.ISO_ERR_ARG
    assert st(cfg(lr=float("nan"))) == _abi.ISO_ERR_ARG
    assert st(cfg(ns_iters=65)) == _abi.ISO_ERR_ARG
    assert st(wsb=1024) == _abi.ISO_ERR_WORKSPACE
    assert st(U=0x100004) == _abi.ISO_ERR_ALIGN
    assert st(mU=0x500002) == _abi.ISO_ERR_ALIGN
    assert st(U=0) == _abi.ISO_ERR_ARG


def test_host_update_sizes_and_argument_errors():
    L = _abi.lib()
    cfg = iso.merge_cfg("iso", 0.05)
    # three 64 x 64 bf16 tensors per list, each list back to back in memory
    th0 = _arr(*[_fake(64, 64, ptr=0x100000 + 8192 * i) for i in range(3)])
    upd = _arr(*[_fake(64, 64, ptr=0x200000 + 8192 * i) for i in range(3)])
    out = _arr(*[_fake(64, 64, ptr=0x300000 + 8192 * i) for i in range(3)])
    nb = ctypes.c_size_t()

    def size(group, cfg_=cfg, n=3):
        rc = L.iso_update_host_staging_size(th0, upd, out, n, ctypes.byref(cfg_), group, ctypes.byref(nb))
        return rc, nb.value

    rc, one_group = size(1 << 30)
    assert rc == 0 and one_group % 256 == 0
    rc, per_tensor = size(1)                       # a group per tensor: slots hold one tensor
    assert rc == 0 and per_tensor < one_group
    assert one_group >= 2 * 3 * 3 * 8192           # two slots of three lists of three tensors
    glob = iso.merge_cfg("ties", 0.2, "global")    # one unit over every tensor: one group
    assert size(1, glob) == size(1 << 30, glob)
    assert size(0)[0] == _abi.ISO_ERR_ARG
    assert L.iso_update_host_staging_size(th0, upd, out, 3, ctypes.byref(cfg), 1 << 20, None) == _abi.ISO_ERR_ARG
    bad_out = _arr(_fake(64, 64, ptr=0x300000), _fake(64, 64, ptr=0x200000), _fake(64, 64, ptr=0x300000 + 16384))
    assert L.iso_update_host_staging_size(th0, upd, bad_out, 3, ctypes.byref(cfg), 1 << 20,
                                          ctypes.byref(nb)) == _abi.ISO_ERR_ARG    # out on an update

    streams = (ctypes.c_void_p * 3)()
    _, need = size(1 << 20)

    def run(staging, nbytes, streams_=streams, n=3, group=1 << 20):
        return L.iso_update_host(th0, upd, 0, out, n, ctypes.byref(cfg), group, ctypes.c_void_p(staging),
                                 nbytes, None, streams_)

    # every rejection happens before anything is enqueued
    assert run(0x4000000, need, streams_=None) == _abi.ISO_ERR_ARG
    assert run(0x4000000, need, group=0) == _abi.ISO_ERR_ARG
    assert run(0, need) == _abi.ISO_ERR_WORKSPACE
    assert run(0x4000010, need) == _abi.ISO_ERR_WORKSPACE                   # not 256-byte aligned
    assert run(0x4000000, need - 256) == _abi.ISO_ERR_WORKSPACE
    assert run(0, 0, n=0) == 0                                              # an empty list is a no-op


def test_range_selection_argument_errors():
    L = _abi.lib()
    x = _arr(_fake(100, 100, ptr=0x100000))
    base = _arr(_fake(100, 100, ptr=0x200000))
    cnt = ctypes.c_void_p(0x300000)

    def hist(b=0, e=10_000, prefix=0, pshift=31, shift=20, nb=2048, counts=cnt, base_=base, x_=x):
        return L.iso_range_hist(x_, base_, b, e, prefix, pshift, shift, nb, counts, None)

    # every rejection happens before anything is enqueued
    assert hist(nb=3) == _abi.ISO_ERR_ARG                      # not a power of two
    assert hist(nb=8192) == _abi.ISO_ERR_ARG
    assert hist(shift=25, pshift=20) == _abi.ISO_ERR_ARG       # shift above pshift
    assert hist(pshift=33) == _abi.ISO_ERR_ARG
    assert hist(b=5, e=4) == _abi.ISO_ERR_ARG
    assert hist(e=10_001) == _abi.ISO_ERR_ARG                  # past the tensor
    assert hist(counts=None) == _abi.ISO_ERR_ARG
    assert hist(base_=_arr(_fake(100, 99, ptr=0x200000))) == _abi.ISO_ERR_SHAPE
    assert hist(x_=_arr(_fake(100, 100, ptr=0x100002))) == _abi.ISO_ERR_ARG      # misaligned
    nb = ctypes.c_size_t()
    assert L.iso_range_mask_workspace_size(10_000, ctypes.byref(nb)) == 0 and nb.value == 10 * 8
    mask = ctypes.c_void_p(0x400000)
    ws = ctypes.c_void_p(0x500000)
    assert L.iso_range_mask(x, base, 0, 10_000, 5, -1, mask, ws, 80, None) == _abi.ISO_ERR_ARG
    assert L.iso_range_mask(x, base, 0, 10_000, 5, 0, mask, ws, 72, None) == _abi.ISO_ERR_WORKSPACE
    assert L.iso_range_mask(x, base, 0, 10_000, 5, 0, mask, None, 80, None) == _abi.ISO_ERR_WORKSPACE
    assert L.iso_range_mask(x, base, 0, 10_000, 5, 0, None, ws, 80, None) == _abi.ISO_ERR_ARG
    assert L.iso_range_mask(x, base, 7, 7, 5, 0, None, None, 0, None) == 0     # an empty range is a no-op
