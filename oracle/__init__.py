"""CPU oracle for the ISO delta-merge hot path -- TEST INFRASTRUCTURE ONLY.

A plain, slow, single-threaded restatement of what the paper
("ISO: An RLVR-Native Optimization Stack") defines for the element-wise merge
path.  The arithmetic lives in ``iso_oracle.c`` (compiled with
``-ffp-contract=off``); this module only gathers the entries of each selection
unit, calls the C routines and scatters the results back.

* task vector ``tau_i = theta_i - theta_0``                       (App. F)
* ``TopKMask(|tau_i|, rho)``, trim ``m_i * tau_i``                 (App. F, TIES)
* TIES: sign election, agreeing set, disjoint mean, ``theta_0 + lambda tau``
                                                                   (App. F)
* Task Arithmetic ``theta_0 + lambda sum_i tau_i``                 (App. F)
* RAM: active set ``|tau_i| > eps_act``, unique values kept, shared ones
  averaged over the active experts                                 (App. F)
* ISO retention combiner (Gram, ridge solve, clip) applied to the trimmed
  task vectors, and the 1-D task-vector average    (Sec. 4.2, App. E, Alg. 1)

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline
leg may import this package.  It shares no code with the CUDA library.

Arrays: bfloat16 tensors are ``numpy.uint16`` bit patterns, binary32 tensors
are ``numpy.float32``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")
_SRC = os.path.join(_HERE, "iso_oracle.c")

BF16, F32 = 0, 1
TA, TIES, ISO, RAM = 0, 1, 2, 3
SCOPE_TENSOR, SCOPE_BLOCK, SCOPE_GLOBAL = 0, 1, 2

KEY_NONE = 0xFFFFFFFF  # threshold key reported for a unit that selects nothing

UNIT_STATS_DTYPE = np.dtype([
    ("thresh_key", np.uint32), ("pad", np.uint32), ("k", np.int64),
    ("count_above", np.int64), ("ties_at_thresh", np.int64), ("ties_taken", np.int64),
])


class _UnitStats(ctypes.Structure):
    _fields_ = [("thresh_key", ctypes.c_uint32), ("pad", ctypes.c_uint32),
                ("k", ctypes.c_int64), ("count_above", ctypes.c_int64),
                ("ties_at_thresh", ctypes.c_int64), ("ties_taken", ctypes.c_int64)]


_lock = threading.Lock()
_handle = None


def build(force: bool = False) -> str:
    """Compile the oracle's C source into ``oracle/_build/liboracle.so``."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < max(
            os.path.getmtime(_SRC), os.path.getmtime(os.path.join(_HERE, "iso_oracle.h"))):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC",
                               "-shared", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _SO)
    return _SO


def _lib():
    global _handle
    with _lock:
        if _handle is None:
            # ISO_ORACLE_LIB lets the mutation tests load a deliberately broken copy
            lib = ctypes.CDLL(os.environ.get("ISO_ORACLE_LIB") or build())
            P = ctypes.c_void_p
            i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            lib.orc_topk_k.restype = i64
            lib.orc_topk_k.argtypes = [f64, i64]
            lib.orc_load.argtypes = [P, i32, i64, P, P]
            lib.orc_delta.argtypes = [P, i32, P, i32, i64, P, P]
            lib.orc_topk_sort.argtypes = [P, i64, i64, P, P]
            lib.orc_topk_select.argtypes = [P, i64, i64, P, P]
            lib.orc_merge_tensor.argtypes = [i32, i32, i64, i32, P, P, P, P,
                                             f64, f64, f64, f64, P, P, P]
            lib.orc_retention.argtypes = [i32, P, f64, f64, f64, P]
            lib.orc_merge_ram.argtypes = [i32, i64, P, P, P, f64, f64, P]
            lib.orc_f64_to_bf16.restype = ctypes.c_uint16
            lib.orc_f64_to_bf16.argtypes = [f64]
            lib.orc_f32_to_bf16.restype = ctypes.c_uint16
            lib.orc_f32_to_bf16.argtypes = [ctypes.c_float]
            lib.orc_f32_to_bf16_array.argtypes = [P, i64, P]
            lib.orc_f64_to_bf16_array.argtypes = [P, i64, P]
            lib.orc_bf16_to_f32.restype = ctypes.c_float
            lib.orc_bf16_to_f32.argtypes = [ctypes.c_uint16]
            _handle = lib
    return _handle


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.uint16:
        return BF16
    if a.dtype == np.float32:
        return F32
    raise TypeError(f"oracle tensors are uint16 (bfloat16 bits) or float32, got {a.dtype}")


# ---------------------------------------------------------------------------
# conversions
# ---------------------------------------------------------------------------

def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    b = np.ascontiguousarray(b, dtype=np.uint16)
    out = np.empty(b.shape, np.float32)
    _lib().orc_load(_ptr(b), BF16, b.size, _ptr(out), None)
    return out


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, np.uint16)
    _lib().orc_f32_to_bf16_array(_ptr(x), x.size, _ptr(out))
    return out


def f64_to_bf16(x: np.ndarray) -> np.ndarray:
    """One rounding from binary64 to bfloat16, ties to even."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    out = np.empty(x.shape, np.uint16)
    _lib().orc_f64_to_bf16_array(_ptr(x), x.size, _ptr(out))
    return out


def to_dtype(values64: np.ndarray, code: int) -> np.ndarray:
    """Round binary64 merge results to the output encoding (once)."""
    if code == F32:
        return np.asarray(values64, dtype=np.float64).astype(np.float32)
    return f64_to_bf16(values64)


# ---------------------------------------------------------------------------
# task vectors and TopKMask
# ---------------------------------------------------------------------------

def k_of(rho: float, n: int) -> int:
    """k = floor(rho n + 1/2) clamped to [0, n]."""
    return int(_lib().orc_topk_k(float(rho), int(n)))


def load(x: np.ndarray):
    """(binary32, binary64) copies of a tensor."""
    x = np.ascontiguousarray(x).ravel()
    v32 = np.empty(x.size, np.float32)
    v64 = np.empty(x.size, np.float64)
    _lib().orc_load(_ptr(x), dtype_code(x), x.size, _ptr(v32), _ptr(v64))
    return v32, v64


def delta(theta_i: np.ndarray, theta_0: np.ndarray):
    """tau = theta_i - theta_0 as (binary32 subtraction, binary64 value)."""
    a = np.ascontiguousarray(theta_i).ravel()
    b = np.ascontiguousarray(theta_0).ravel()
    if a.size != b.size:
        raise ValueError("shape mismatch")
    tau32 = np.empty(a.size, np.float32)
    tau64 = np.empty(a.size, np.float64)
    _lib().orc_delta(_ptr(a), dtype_code(a), _ptr(b), dtype_code(b), a.size,
                     _ptr(tau32), _ptr(tau64))
    return tau32, tau64


def topk_unit(tau32: np.ndarray, k: int, method: str = "select"):
    """TopKMask over one unit given in unit order; returns (mask, stats row)."""
    t = np.ascontiguousarray(tau32, dtype=np.float32)
    mask = np.empty(t.size, np.uint8)
    st = _UnitStats()
    fn = _lib().orc_topk_select if method == "select" else _lib().orc_topk_sort
    fn(_ptr(t), t.size, int(k), _ptr(mask), ctypes.byref(st))
    row = np.zeros((), UNIT_STATS_DTYPE)
    for name, _ in _UnitStats._fields_:
        row[name] = getattr(st, name)
    return mask, row


def block_units(rows: int, cols: int, br: int, bc: int):
    """Flat indices of each br x bc block of a row-major rows x cols tensor,
    blocks in row-major block order, entries row-major inside a block (this is
    the tensor's own index order restricted to the block).  Edge blocks are
    partial."""
    out = []
    for r0 in range(0, rows, br):
        r = np.arange(r0, min(rows, r0 + br), dtype=np.int64)
        for c0 in range(0, cols, bc):
            c = np.arange(c0, min(cols, c0 + bc), dtype=np.int64)
            out.append((r[:, None] * cols + c[None, :]).ravel())
    return out


def topk_masks(tau32_list, shapes, density, scope=SCOPE_TENSOR, block=(128, 128),
               method="select", participate=None):
    """TopKMask of one task vector given as a list of tensors.

    ``participate[t]`` False leaves tensor t unmasked (its units report k = -1).
    Returns (masks per tensor, unit stats array in the unit order used by the
    library: tensor order, and row-major block order inside a tensor).
    """
    n_t = len(tau32_list)
    if participate is None:
        participate = [True] * n_t
    masks = [np.zeros(np.asarray(t).size, np.uint8) for t in tau32_list]
    stats = []

    def skipped_row():
        row = np.zeros((), UNIT_STATS_DTYPE)
        row["thresh_key"] = KEY_NONE
        row["k"] = -1
        return row

    if scope == SCOPE_GLOBAL:
        if not any(participate):
            return masks, np.array([skipped_row()], UNIT_STATS_DTYPE)
        parts = [np.asarray(tau32_list[t], np.float32).ravel() for t in range(n_t) if participate[t]]
        cat = np.concatenate(parts) if parts else np.zeros(0, np.float32)
        m, row = topk_unit(cat, k_of(density, cat.size), method)
        off = 0
        for t in range(n_t):
            if participate[t]:
                n = masks[t].size
                masks[t][:] = m[off:off + n]
                off += n
        return masks, np.array([row], UNIT_STATS_DTYPE)

    for t in range(n_t):
        tau = np.asarray(tau32_list[t], np.float32).ravel()
        rows, cols = shapes[t]
        if scope == SCOPE_TENSOR:
            if participate[t]:
                m, row = topk_unit(tau, k_of(density, tau.size), method)
                masks[t][:] = m
                stats.append(row)
            else:
                stats.append(skipped_row())
        else:
            for idx in block_units(rows, cols, block[0], block[1]):
                if participate[t]:
                    m, row = topk_unit(tau[idx], k_of(density, idx.size), method)
                    masks[t][idx] = m
                    stats.append(row)
                else:
                    stats.append(skipped_row())
    return masks, np.array(stats, UNIT_STATS_DTYPE)


# ---------------------------------------------------------------------------
# merge / update
# ---------------------------------------------------------------------------

def retention(gram: np.ndarray, ridge=1e-12, c_min=0.0, c_max=1.5) -> np.ndarray:
    g = np.ascontiguousarray(gram, dtype=np.float64)
    K = g.shape[0]
    c = np.zeros(K, np.float64)
    _lib().orc_retention(K, _ptr(g), ridge, c_min, c_max, _ptr(c))
    return c


def merge(theta0, experts, op, *, experts_are_deltas=True, density=0.2,
          scope=SCOPE_TENSOR, block=(128, 128), lam=1.0, ridge=1e-12, c_min=0.0,
          c_max=1.5, mask_1d=True, shapes=None, is_1d=None, method="select",
          eps_act=float(np.float32(1e-5))):
    """Merge K experts into the base, tensor by tensor.

    theta0       list of base tensors (uint16 bfloat16 bits or float32)
    experts      list of K lists of tensors: task vectors (experts_are_deltas)
                 or fine-tuned checkpoints
    op           TA / TIES / ISO / RAM
    eps_act      RAM activity threshold; the default is the paper's 1e-5 as
                 a binary32 value (the library takes the threshold in binary32)
    shapes       list of (rows, cols); defaults to each array's 2-D shape
    is_1d        list of flags; defaults to rows == 1 for 1-row tensors

    Returns a dict: ``out`` (tensors in the base encoding), ``out64`` (binary64
    values before the final rounding), ``mag`` (per-entry |theta_0| + sum of the
    magnitudes of the update terms, used for tolerances), ``units`` (K x
    n_units stats), ``gram`` and ``coef`` (per tensor, ISO only).
    """
    lib = _lib()
    K = len(experts)
    n_t = len(theta0)
    if shapes is None:
        shapes = [(a.shape[0], a.shape[1]) if a.ndim == 2 else (1, a.size) for a in theta0]
    if is_1d is None:
        is_1d = [np.asarray(a).ndim == 1 for a in theta0]
    tau32 = [[None] * n_t for _ in range(K)]
    tau64 = [[None] * n_t for _ in range(K)]
    for i in range(K):
        for t in range(n_t):
            if experts_are_deltas:
                tau32[i][t], tau64[i][t] = load(experts[i][t])
            else:
                tau32[i][t], tau64[i][t] = delta(experts[i][t], theta0[t])

    if op in (TA, RAM):
        participate = [False] * n_t
    elif op == TIES:
        participate = [True if mask_1d else not is_1d[t] for t in range(n_t)]
    else:
        participate = [not is_1d[t] for t in range(n_t)]

    masks = [None] * K
    units = []
    if op not in (TA, RAM):   # every trimming operator reports one row per unit (k = -1: not trimmed)
        for i in range(K):
            masks[i], st = topk_masks(tau32[i], shapes, density, scope, block, method, participate)
            units.append(st)
    out, out64, mag, grams, coefs = [], [], [], [], []
    for t in range(n_t):
        n = np.asarray(theta0[t]).size
        th32, th64 = load(theta0[t])
        o64 = np.empty(n, np.float64)
        g = np.zeros((K, K), np.float64)
        c = np.zeros(K, np.float64)
        t32 = [np.ascontiguousarray(tau32[i][t]) for i in range(K)]
        t64 = [np.ascontiguousarray(tau64[i][t]) for i in range(K)]
        P32 = (ctypes.c_void_p * K)(*[a.ctypes.data for a in t32])
        P64 = (ctypes.c_void_p * K)(*[a.ctypes.data for a in t64])
        use_mask = participate[t] and op not in (TA, RAM)
        if use_mask:
            mk = [np.ascontiguousarray(masks[i][t]) for i in range(K)]
            PM = (ctypes.c_void_p * K)(*[a.ctypes.data for a in mk])
        else:
            mk = None
            PM = None
        if op == RAM:
            lib.orc_merge_ram(K, n, _ptr(th64), P32, P64, float(eps_act), float(lam), _ptr(o64))
        else:
            lib.orc_merge_tensor(op, K, n, int(bool(is_1d[t])), _ptr(th64), P32, P64, PM,
                                 float(lam), float(ridge), float(c_min), float(c_max),
                                 _ptr(o64), _ptr(g), _ptr(c))
        code = dtype_code(np.asarray(theta0[t]))
        out.append(to_dtype(o64, code).reshape(np.shape(theta0[t])))
        out64.append(o64)
        m = np.abs(th64).copy()
        for i in range(K):
            term = np.abs(t64[i])
            if use_mask:
                term = term * mk[i]
            if op == ISO and not is_1d[t]:
                term = term * abs(c[i])
            elif op == ISO:
                term = term / K
            else:
                term = term * abs(lam)
            m += term
        mag.append(m)
        grams.append(g)
        coefs.append(c)
    return {"out": out, "out64": out64, "mag": mag, "masks": masks,
            "units": np.stack(units) if units else np.zeros((0, 0), UNIT_STATS_DTYPE),
            "gram": grams, "coef": coefs}


def update(theta0, update_tensors, op=ISO, *, update_is_delta=False, **kw):
    """The K = 1 masked update: ``merge`` with one expert."""
    return merge(theta0, [update_tensors], op, experts_are_deltas=update_is_delta, **kw)
