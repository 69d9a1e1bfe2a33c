"""PyTorch-facing binding of the C ABI (include/iso.h).

Argument marshalling only: every function here builds the ABI descriptors
from ``torch.Tensor`` objects (device memory and streams come from PyTorch)
and calls the entry point of the same name in libiso_gb300.so, where every
step of the computation runs.  There is no CPU path.
"""
from __future__ import annotations

import ctypes
from dataclasses import dataclass
from typing import List, Optional, Sequence

import numpy as np
import torch

from . import _abi
from ._abi import (IsoMergeCfg, IsoMergeStats, IsoTensor, IsoTopkCfg, check, lib)

OPS = {"ta": _abi.ISO_OP_TA, "ties": _abi.ISO_OP_TIES, "iso": _abi.ISO_OP_ISO, "ram": _abi.ISO_OP_RAM}
SCOPES = {"tensor": _abi.ISO_SCOPE_TENSOR, "block": _abi.ISO_SCOPE_BLOCK,
          "global": _abi.ISO_SCOPE_GLOBAL}
UNIT_STATS_DTYPE = np.dtype([
    ("thresh_key", np.uint32), ("flags", np.uint32), ("k", np.int64),
    ("count_above", np.int64), ("ties_at_thresh", np.int64), ("ties_taken", np.int64),
])
assert UNIT_STATS_DTYPE.itemsize == ctypes.sizeof(_abi.IsoUnitStats)


def _code(dtype: torch.dtype) -> int:
    if dtype == torch.bfloat16:
        return _abi.ISO_BF16
    if dtype == torch.float32:
        return _abi.ISO_F32
    raise TypeError(f"tensors must be bfloat16 or float32, got {dtype}")


def _shape2d(t: torch.Tensor):
    if t.dim() == 2:
        return int(t.shape[0]), int(t.shape[1]), 0
    if t.dim() == 1:
        return 1, int(t.shape[0]), 1
    raise ValueError("tensors must be 1-D or 2-D")


def describe(ts: Sequence[torch.Tensor], is_1d: Optional[Sequence[bool]] = None):
    """ctypes array of iso_tensor for a list of contiguous tensors."""
    arr = (IsoTensor * max(1, len(ts)))()
    for q, t in enumerate(ts):
        if not t.is_contiguous():
            raise ValueError("tensors must be contiguous")
        r, c, one = _shape2d(t)
        if is_1d is not None:
            one = int(bool(is_1d[q]))
        arr[q] = IsoTensor(t.data_ptr() if t.numel() else None, r, c, _code(t.dtype), one)
    return arr


def topk_cfg(density=0.05, scope="tensor", block=(128, 128)) -> IsoTopkCfg:
    return IsoTopkCfg(float(density), SCOPES[scope], int(block[0]), int(block[1]), 0)


def merge_cfg(op="ties", density=0.2, scope="tensor", block=(128, 128), lam=1.0, ridge=1e-12,
              c_min=0.0, c_max=1.5, mask_1d=True, eps_act=1e-5) -> IsoMergeCfg:
    """eps_act (RAM) is passed as a binary32 value."""
    return IsoMergeCfg(OPS[op], int(bool(mask_1d)), float(lam), float(eps_act), float(ridge),
                       float(c_min), float(c_max), topk_cfg(density, scope, block))


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


@dataclass
class Stats:
    """Device-side outputs of one call (see iso_merge_stats)."""
    status: torch.Tensor          # int32[1]
    units: torch.Tensor           # uint8[K * n_units * 40]
    gram: Optional[torch.Tensor]  # float64[n_tensors * K * K]
    coef: Optional[torch.Tensor]  # float64[n_tensors * K]
    K: int
    n_units: int

    def abi(self) -> IsoMergeStats:
        return IsoMergeStats(self.status.data_ptr(), self.units.data_ptr(),
                             self.gram.data_ptr() if self.gram is not None else None,
                             self.coef.data_ptr() if self.coef is not None else None)

    def units_numpy(self) -> np.ndarray:
        raw = self.units.cpu().numpy()
        return raw.view(UNIT_STATS_DTYPE).reshape(self.K, self.n_units)


def make_stats(tensors, K, topk: IsoTopkCfg, device, with_gram=True) -> Stats:
    n_units = iso_num_units(tensors, topk)
    n = len(tensors)
    return Stats(
        status=torch.zeros(1, dtype=torch.int32, device=device),
        units=torch.zeros(max(1, K * n_units) * UNIT_STATS_DTYPE.itemsize, dtype=torch.uint8, device=device),
        gram=torch.zeros(max(1, n * K * K), dtype=torch.float64, device=device) if with_gram else None,
        coef=torch.zeros(max(1, n * K), dtype=torch.float64, device=device) if with_gram else None,
        K=K, n_units=n_units)


class Workspace:
    """Caller-owned scratch for the library, one growing torch buffer."""

    def __init__(self, device=None):
        self.device = torch.device(device or "cuda")
        self.buf = torch.empty(0, dtype=torch.uint8, device=self.device)

    def get(self, nbytes: int):
        if self.buf.numel() < nbytes:
            self.buf = torch.empty(nbytes + 256, dtype=torch.uint8, device=self.device)
        ptr = self.buf.data_ptr()
        off = (-ptr) % 256
        return ctypes.c_void_p(ptr + off), self.buf.numel() - off


_default_ws = {}


def _workspace(ws: Optional[Workspace], device) -> Workspace:
    if ws is not None:
        return ws
    key = torch.device(device).index
    if key not in _default_ws:
        _default_ws[key] = Workspace(device)
    return _default_ws[key]


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------

def iso_num_units(tensors, topk: IsoTopkCfg) -> int:
    d = describe(tensors)
    n = ctypes.c_int64(0)
    check(lib().iso_num_units(d, len(tensors), ctypes.byref(topk), ctypes.byref(n)), "iso_num_units")
    return int(n.value)


def iso_workspace_size(tensors, K: int, cfg: IsoMergeCfg):
    """(minimum, full) workspace bytes."""
    d = describe(tensors)
    mn, full = ctypes.c_size_t(0), ctypes.c_size_t(0)
    check(lib().iso_workspace_size(d, len(tensors), int(K), ctypes.byref(cfg), ctypes.byref(mn),
                                   ctypes.byref(full)), "iso_workspace_size")
    return int(mn.value), int(full.value)


def iso_delta(theta_i: List[torch.Tensor], theta_0: List[torch.Tensor], tau=None, stream=None):
    if tau is None:
        tau = [torch.empty(t.shape, dtype=torch.float32, device=t.device) for t in theta_0]
    check(lib().iso_delta(describe(theta_i), describe(theta_0), describe(tau), len(theta_0),
                          _stream(stream)), "iso_delta")
    return tau


def iso_topk_mask(tau: List[torch.Tensor], density=0.2, scope="tensor", block=(128, 128),
                  masks=None, workspace: Optional[Workspace] = None, stats=False, stream=None,
                  ws_bytes: Optional[int] = None):
    """Packed TopKMask of a task vector: per tensor ceil(numel/32) int32 words."""
    dev = tau[0].device
    cfg = topk_cfg(density, scope, block)
    if masks is None:
        masks = [torch.zeros((t.numel() + 31) // 32 + 4, dtype=torch.int32, device=dev) for t in tau]
    mptrs = (ctypes.c_void_p * max(1, len(tau)))(*[m.data_ptr() for m in masks])
    mcfg = merge_cfg("ties", density, scope, block)
    _, full = iso_workspace_size(tau, 1, mcfg)
    ws = _workspace(workspace, dev)
    wptr, wlen = ws.get(full if ws_bytes is None else ws_bytes)
    st = make_stats(tau, 1, cfg, dev, with_gram=False) if stats else None
    check(lib().iso_topk_mask(describe(tau), len(tau), ctypes.byref(cfg), mptrs,
                              ctypes.byref(st.abi()) if st else None, wptr,
                              wlen if ws_bytes is None else ws_bytes, _stream(stream)),
          "iso_topk_mask")
    out = [m[: (t.numel() + 31) // 32] for m, t in zip(masks, tau)]
    return (out, st) if stats else out


def iso_merge(theta_0: List[torch.Tensor], experts: List[List[torch.Tensor]], op="ties",
              experts_are_deltas=True, out=None, density=0.2, scope="tensor", block=(128, 128),
              lam=1.0, ridge=1e-12, c_min=0.0, c_max=1.5, mask_1d=True, is_1d=None,
              workspace: Optional[Workspace] = None, stats=False, stream=None,
              ws_bytes: Optional[int] = None, eps_act=1e-5):
    """Merge K experts into the base (iso_merge; iso_update for K = 1).

    op is "ta", "ties", "iso" or "ram"; experts holds K lists of tensors
    shaped like theta_0 (task vectors, or checkpoints when
    experts_are_deltas is False).  density / scope / block configure the
    TopKMask of TIES and ISO; lam scales TA, TIES and RAM; ridge / c_min /
    c_max configure ISO's retention solve; eps_act is RAM's activity
    threshold.  Returns the outputs (and the device-side stats when
    stats=True)."""
    K = len(experts)
    n = len(theta_0)
    dev = theta_0[0].device
    if out is None:
        out = [torch.empty_like(t) for t in theta_0]
    cfg = merge_cfg(op, density, scope, block, lam, ridge, c_min, c_max, mask_1d, eps_act)
    flat = [x for e in experts for x in e]
    d0 = describe(theta_0, is_1d)
    dx = describe(flat, None if is_1d is None else list(is_1d) * K)
    do = describe(out, is_1d)
    _, full = iso_workspace_size(theta_0, K, cfg)
    ws = _workspace(workspace, dev)
    wptr, wlen = ws.get(full if ws_bytes is None else ws_bytes)
    st = make_stats(theta_0, K, cfg.topk, dev) if stats else None
    fn = lib().iso_update if K == 1 else None
    if K == 1:
        rc = fn(d0, dx, int(bool(experts_are_deltas)), do, n, ctypes.byref(cfg), wptr,
                wlen if ws_bytes is None else ws_bytes, ctypes.byref(st.abi()) if st else None,
                _stream(stream))
        check(rc, "iso_update")
    else:
        rc = lib().iso_merge(d0, dx, K, int(bool(experts_are_deltas)), do, n, ctypes.byref(cfg),
                             wptr, wlen if ws_bytes is None else ws_bytes,
                             ctypes.byref(st.abi()) if st else None, _stream(stream))
        check(rc, "iso_merge")
    return (out, st) if stats else out


def iso_update(theta_0: List[torch.Tensor], update: List[torch.Tensor], op="iso",
               update_is_delta=False, **kw):
    """The K = 1 masked update (iso_update)."""
    return iso_merge(theta_0, [update], op=op, experts_are_deltas=update_is_delta, **kw)


def iso_update_host_staging_size(theta_0, update, out, op="iso", density=0.05, scope="tensor",
                                 block=(128, 128), lam=1.0, ridge=1e-12, c_min=0.0, c_max=1.5,
                                 mask_1d=True, eps_act=1e-5, group_bytes=2 << 30) -> int:
    cfg = merge_cfg(op, density, scope, block, lam, ridge, c_min, c_max, mask_1d, eps_act)
    nb = ctypes.c_size_t(0)
    check(lib().iso_update_host_staging_size(describe(theta_0), describe(update), describe(out),
                                              len(theta_0), ctypes.byref(cfg), int(group_bytes),
                                              ctypes.byref(nb)), "iso_update_host_staging_size")
    return int(nb.value)


class HostUpdate:
    """The K = 1 update of tensors in host memory (iso_update_host): groups of
    tensors are copied in, updated and copied back in a pipeline over three
    CUDA streams.  Host tensors should be page-locked (pin_memory) for the
    copies to overlap the update; out may be the theta_0 tensors themselves."""

    def __init__(self, device="cuda", group_bytes=2 << 30):
        self.dev = torch.device(device)
        self.group_bytes = int(group_bytes)
        self.streams = [torch.cuda.Stream(self.dev) for _ in range(3)]
        self.ws = Workspace(self.dev)
        self.h2d_bytes = self.d2h_bytes = 0

    def run(self, theta_0, update, out=None, op="iso", update_is_delta=False, density=0.05,
            scope="tensor", block=(128, 128), lam=1.0, ridge=1e-12, c_min=0.0, c_max=1.5, mask_1d=True,
            eps_act=1e-5, stats=False, stream=None):
        """Enqueue the update; it has finished once ``stream`` (default: the
        current stream) reaches the point where this call returned."""
        if out is None:
            out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in theta_0]
        cfg = merge_cfg(op, density, scope, block, lam, ridge, c_min, c_max, mask_1d, eps_act)
        d0, d1, do = describe(theta_0), describe(update), describe(out)
        nb = ctypes.c_size_t(0)
        check(lib().iso_update_host_staging_size(d0, d1, do, len(theta_0), ctypes.byref(cfg),
                                                  self.group_bytes, ctypes.byref(nb)),
              "iso_update_host_staging_size")
        wptr, wlen = self.ws.get(int(nb.value))
        st = make_stats(theta_0, 1, cfg.topk, self.dev) if stats else None
        cur = stream if stream is not None else torch.cuda.current_stream(self.dev)
        h2d, comp, d2h = self.streams
        # the pipeline starts after the caller's earlier work and ends on the
        # caller's stream
        for s_ in self.streams:
            s_.wait_stream(cur)
        ptrs = (ctypes.c_void_p * 3)(h2d.cuda_stream, comp.cuda_stream, d2h.cuda_stream)
        check(lib().iso_update_host(d0, d1, int(bool(update_is_delta)), do, len(theta_0),
                                    ctypes.byref(cfg), self.group_bytes, wptr, wlen,
                                    ctypes.byref(st.abi()) if st else None, ptrs), "iso_update_host")
        cur.wait_stream(comp)
        self.h2d_bytes = sum(t.numel() * t.element_size() for t in list(theta_0) + list(update))
        self.d2h_bytes = sum(t.numel() * t.element_size() for t in out)
        return (out, st) if stats else out


# ---------------------------------------------------------------------------
# one selection unit split over ranks (App. F, TIES trim)
# ---------------------------------------------------------------------------
def _range_args(x, base, begin, end):
    n = x.numel()
    end = n if end is None else int(end)
    dx = describe([x])
    db = describe([base]) if base is not None else None
    return dx, db, int(begin), end


def range_hist(x: torch.Tensor, base: Optional[torch.Tensor] = None, begin=0, end=None, prefix=0, pshift=32,
               shift=21, nbins=2048, counts=None, stream=None) -> torch.Tensor:
    """iso_range_hist: int64[nbins] device counts of the magnitude keys of
    x[begin:end] (x - base for a checkpoint) with key >> pshift == prefix,
    binned by (key >> shift) & (nbins - 1)."""
    dx, db, b, e = _range_args(x, base, begin, end)
    if counts is None:
        counts = torch.empty(nbins, dtype=torch.int64, device=x.device)
    check(lib().iso_range_hist(dx, db, b, e, int(prefix) & 0xFFFFFFFF, int(pshift), int(shift), int(nbins),
                               ctypes.c_void_p(counts.data_ptr()), _stream(stream)), "iso_range_hist")
    return counts


def range_mask(x: torch.Tensor, t: int, take: int, base: Optional[torch.Tensor] = None, begin=0, end=None,
               workspace: Optional[Workspace] = None, stream=None) -> torch.Tensor:
    """iso_range_mask: packed int32 words of this range's share of a unit's
    TopKMask (keys above t, and the first ``take`` keys equal to t)."""
    dx, db, b, e = _range_args(x, base, begin, end)
    words = torch.zeros(max(1, (e - b + 31) // 32), dtype=torch.int32, device=x.device)
    nb = ctypes.c_size_t(0)
    check(lib().iso_range_mask_workspace_size(e - b, ctypes.byref(nb)), "iso_range_mask_workspace_size")
    ws = _workspace(workspace, x.device)
    wptr, wlen = ws.get(int(nb.value))
    check(lib().iso_range_mask(dx, db, b, e, int(t) & 0xFFFFFFFF, int(take), ctypes.c_void_p(words.data_ptr()),
                               wptr, wlen, _stream(stream)), "iso_range_mask")
    return words[: (e - b + 31) // 32]


def split_unit_topk(x: torch.Tensor, density: float, base: Optional[torch.Tensor] = None, begin=0, end=None,
                    group=None, workspace: Optional[Workspace] = None):
    """This rank's part of the exact TopKMask of one unit split over the ranks
    of ``group`` (rank order = position order): the radix counts come from
    iso_range_hist on the device, summed over the ranks by
    shard.split_unit_select; the mask words from iso_range_mask.  Returns
    (SplitSelect, int32 mask words of x[begin:end])."""
    from .shard import split_unit_select
    dx, db, b, e = _range_args(x, base, begin, end)

    def local_hist(prefix, pshift, shift, nb):
        return range_hist(x, base, b, e, prefix, pshift, shift, nb).cpu().tolist()

    def local_ties(t):
        return int(range_hist(x, base, b, e, t, 0, 0, 1).cpu()[0])

    sel = split_unit_select(e - b, density, local_hist, local_ties, group=group)
    return sel, range_mask(x, sel.t, sel.take, base, b, e, workspace=workspace)


def launch_count() -> int:
    return int(lib().iso_launch_count())


def force_two_pass(on=True):
    """Diagnostics: run later K = 1 updates in the two-pass form."""
    check(lib().iso_force_two_pass(int(bool(on))), "iso_force_two_pass")


def compact_candidates(on=True):
    """Diagnostics: let later K >= 2 TIES / ISO merges read compact candidate
    values in their Gram and merge passes, or the full task vectors (the
    default); the results are the same."""
    check(lib().iso_compact_candidates(int(bool(on))), "iso_compact_candidates")


def profile_enable(on=True):
    check(lib().iso_profile_enable(int(bool(on))), "iso_profile_enable")


def profile_reset():
    check(lib().iso_profile_reset(), "iso_profile_reset")


def profile_read():
    """{kernel kind: (launches, total ms)} since the last reset."""
    res = {}
    for k in range(lib().iso_profile_kinds()):
        n, ms = ctypes.c_int64(0), ctypes.c_double(0.0)
        check(lib().iso_profile_read(k, ctypes.byref(n), ctypes.byref(ms)), "iso_profile_read")
        if n.value:
            res[lib().iso_profile_name(k).decode()] = (int(n.value), float(ms.value))
    return res


def iso_update_noalloc(theta_0: List[torch.Tensor], update: List[torch.Tensor], op="iso",
                       update_is_delta=False, out=None, density=0.05, scope="tensor",
                       block=(128, 128), lam=1.0, ridge=1e-12, c_min=0.0, c_max=1.5,
                       mask_1d=True, stats=False, stream=None, eps_act=1e-5):
    """iso_update for callers that cannot allocate device memory: the library
    runs the update in its own fixed per-device scratch (no workspace
    argument).  Make the first call on a device before any stream capture;
    calls that overlap on the GPU race on the shared scratch."""
    dev = theta_0[0].device
    if out is None:
        out = [torch.empty_like(t) for t in theta_0]
    cfg = merge_cfg(op, density, scope, block, lam, ridge, c_min, c_max, mask_1d, eps_act)
    st = make_stats(theta_0, 1, cfg.topk, dev) if stats else None
    check(lib().iso_update_noalloc(describe(theta_0), describe(update), int(bool(update_is_delta)),
                                   describe(out), len(theta_0), ctypes.byref(cfg),
                                   ctypes.byref(st.abi()) if st else None, _stream(stream)),
          "iso_update_noalloc")
    return (out, st) if stats else out


# ---------------------------------------------------------------------------
# frame-space ISO-Merger of one matrix (App. E)
# ---------------------------------------------------------------------------
@dataclass
class FrameStats:
    """Device-side outputs of iso_frame_merge."""
    status: torch.Tensor   # int32[1]
    gram: torch.Tensor     # float64[K, K]
    coef: torch.Tensor     # float64[K]

    def abi(self) -> IsoMergeStats:
        return IsoMergeStats(self.status.data_ptr(), None, self.gram.data_ptr(), self.coef.data_ptr())


def frame_workspace_size(m: int, n: int, K: int) -> int:
    b = ctypes.c_size_t(0)
    check(lib().iso_frame_workspace_size(int(m), int(n), int(K), ctypes.byref(b)), "iso_frame_workspace_size")
    return int(b.value)


def frame_merge_factors(U0, S0, Vt0, Us, Vts, W0, out=None, rho_keep=0.9, ridge=1e-12, c_min=0.0, c_max=1.5,
                        ns_iters=0, workspace=None, stats=False, stream=None):
    """iso_frame_merge: the ISO-Merger of one m x n matrix from the thin SVD
    factors of the base (U0 m x q, S0 q, Vt0 q x n) and of the K experts (Us,
    Vts), binary64 and contiguous on the device; W0 is the base matrix (bf16
    or fp32).  Returns out (and FrameStats with stats=True)."""
    m, n = int(W0.shape[0]), int(W0.shape[1])
    K = len(Us)
    if len(Vts) != K:
        raise ValueError("one U and one Vt per expert")
    for t in [U0, S0, Vt0, *Us, *Vts]:
        if t.dtype != torch.float64 or not t.is_contiguous():
            raise ValueError("SVD factors must be contiguous float64 tensors")
    if out is None:
        out = torch.empty_like(W0)
    dev = W0.device
    cfg = _abi.IsoFrameCfg(float(rho_keep), float(ridge), float(c_min), float(c_max), int(ns_iters), 0)
    need = frame_workspace_size(m, n, K)
    ws = _workspace(workspace, dev)
    wptr, wlen = ws.get(need)
    up = (ctypes.c_void_p * K)(*[u.data_ptr() for u in Us])
    vp = (ctypes.c_void_p * K)(*[v.data_ptr() for v in Vts])
    st = None
    if stats:
        st = FrameStats(torch.zeros(1, dtype=torch.int32, device=dev),
                        torch.zeros(K, K, dtype=torch.float64, device=dev),
                        torch.zeros(K, dtype=torch.float64, device=dev))
    rc = lib().iso_frame_merge(U0.data_ptr(), S0.data_ptr(), Vt0.data_ptr(), up, vp, K, m, n,
                               describe([W0]), describe([out]), ctypes.byref(cfg), wptr, wlen,
                               ctypes.byref(st.abi()) if st else None, _stream(stream))
    check(rc, "iso_frame_merge")
    return (out, st) if stats else out


def thin_svd(W: torch.Tensor):
    """The thin SVD W = U diag(S) Vt in binary64 on W's device (the library
    SVD of torch.linalg; the frame merge's one step that is not this
    library's own code)."""
    _load_torch_linalg()
    U, S, Vt = torch.linalg.svd(W.to(torch.float64), full_matrices=False)
    return U.contiguous(), S.contiguous(), Vt.contiguous()


def _load_torch_linalg():
    """torch opens its GPU linear-algebra library lazily by name; under a
    profiler that rewrites the library search path that lookup fails, so it is
    loaded once here by its full path when the file is present."""
    import os
    lib_dir = os.path.join(os.path.dirname(torch.__file__), "lib")
    path = os.path.join(lib_dir, "libtorch_cuda_linalg.so")
    if os.path.exists(path) and not getattr(_load_torch_linalg, "done", False):
        ctypes.CDLL(path, mode=ctypes.RTLD_GLOBAL)
        _load_torch_linalg.done = True


def frame_merge(W0: torch.Tensor, experts: Sequence[torch.Tensor], **kw):
    """ISO-Merger of one matrix from the base and K expert checkpoints: the
    thin SVDs (thin_svd), then iso_frame_merge."""
    U0, S0, Vt0 = thin_svd(W0)
    Us, Vts = [], []
    for E in experts:
        U, _, Vt = thin_svd(E)
        Us.append(U)
        Vts.append(Vt)
    return frame_merge_factors(U0, S0, Vt0, Us, Vts, W0, **kw)


def gemm_tf32(A: torch.Tensor, B: torch.Tensor, C: torch.Tensor, Kc: int, a_k0=0, b_k0=0, stream=None):
    """iso_gemm_tf32: C = A[:, a_k0:a_k0+Kc] B[:, b_k0:b_k0+Kc]^T on the tensor cores (tf32)."""
    for t in (A, B, C):
        if t.dtype != torch.float32 or not t.is_contiguous() or t.dim() != 2:
            raise ValueError("gemm_tf32 takes contiguous 2-D float32 tensors")
    rc = lib().iso_gemm_tf32(A.data_ptr(), A.shape[1], B.data_ptr(), B.shape[1], C.data_ptr(), C.shape[1],
                             A.shape[0], B.shape[0], int(Kc), int(a_k0), int(b_k0), _stream(stream))
    check(rc, "iso_gemm_tf32")
    return C


# ---------------------------------------------------------------------------
# ISO-Optimizer step ISO[AdamW] on one matrix (Sec. 4.3)
# ---------------------------------------------------------------------------
def opt_workspace_size(m: int, n: int) -> int:
    b = ctypes.c_size_t(0)
    check(lib().iso_opt_workspace_size(int(m), int(n), ctypes.byref(b)), "iso_opt_workspace_size")
    return int(b.value)


def opt_step(U, V, S0, G_W, mU, vU, mV, vV, W, W_out=None, lr=1e-6, beta1=0.9, beta2=0.999, eps=1e-8,
             weight_decay=0.0, step=1, ns_iters=0, workspace=None, stats=False, stream=None):
    """iso_opt_step: one ISO[AdamW] step of an m x n matrix.  U (m x q) and V
    (n x q) are contiguous float64 frames and mU, vU, mV, vV float32 moments
    of the same shapes, all updated in place; S0 (q) float64; G_W, W (m x n,
    bf16 or fp32).  Returns W_out (and a status tensor with stats=True)."""
    m, n = int(W.shape[0]), int(W.shape[1])
    for t in (U, V, S0):
        if t.dtype != torch.float64 or not t.is_contiguous():
            raise ValueError("frames and spectrum must be contiguous float64 tensors")
    for t in (mU, vU, mV, vV):
        if t.dtype != torch.float32 or not t.is_contiguous():
            raise ValueError("moments must be contiguous float32 tensors")
    if W_out is None:
        W_out = torch.empty_like(W)
    cfg = _abi.IsoAdamwCfg(float(lr), float(beta1), float(beta2), float(eps), float(weight_decay), int(step),
                           int(ns_iters), 0)
    ws = _workspace(workspace, W.device)
    wptr, wlen = ws.get(opt_workspace_size(m, n))
    st = torch.zeros(1, dtype=torch.int32, device=W.device) if stats else None
    abi_st = IsoMergeStats(st.data_ptr(), None, None, None) if stats else None
    rc = lib().iso_opt_step(U.data_ptr(), V.data_ptr(), S0.data_ptr(), describe([G_W]), mU.data_ptr(),
                            vU.data_ptr(), mV.data_ptr(), vV.data_ptr(), describe([W]), describe([W_out]), m, n,
                            ctypes.byref(cfg), wptr, wlen, ctypes.byref(abi_st) if stats else None, _stream(stream))
    check(rc, "iso_opt_step")
    return (W_out, st) if stats else W_out
