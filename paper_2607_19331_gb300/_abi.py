"""ctypes mirror of include/iso.h and the loader of libiso_gb300.so.

This module only describes the C ABI; it performs no computation.  Loading
fails loudly when the shared library has not been built.
"""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "_build", "libiso_gb300.so")

ISO_OK = 0
ISO_ERR_ARG = -1
ISO_ERR_SHAPE = -2
ISO_ERR_DTYPE = -3
ISO_ERR_ALIGN = -4
ISO_ERR_WORKSPACE = -5
ISO_ERR_CUDA = -6
ISO_ERR_NONFINITE = -7
ISO_ERR_UNSUPPORTED = -8
ISO_ERR_TIMEOUT = -9
ISO_MAX_EXPERTS = 8
ISO_NOALLOC_SCRATCH_BYTES = 32 << 20

ISO_BF16, ISO_F32 = 0, 1
ISO_SCOPE_TENSOR, ISO_SCOPE_BLOCK, ISO_SCOPE_GLOBAL = 0, 1, 2
ISO_OP_TA, ISO_OP_TIES, ISO_OP_ISO, ISO_OP_RAM = 0, 1, 2, 3


class IsoTensor(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("is_1d", ctypes.c_int32)]


class IsoTopkCfg(ctypes.Structure):
    _fields_ = [("density", ctypes.c_double), ("scope", ctypes.c_int32),
                ("block_rows", ctypes.c_int32), ("block_cols", ctypes.c_int32),
                ("reserved", ctypes.c_int32)]


class IsoMergeCfg(ctypes.Structure):
    _fields_ = [("op", ctypes.c_int32), ("mask_1d", ctypes.c_int32), ("lam", ctypes.c_float),
                ("eps_act", ctypes.c_float), ("ridge", ctypes.c_double),
                ("c_min", ctypes.c_double), ("c_max", ctypes.c_double), ("topk", IsoTopkCfg)]


class IsoUnitStats(ctypes.Structure):
    _fields_ = [("thresh_key", ctypes.c_uint32), ("flags", ctypes.c_uint32), ("k", ctypes.c_int64),
                ("count_above", ctypes.c_int64), ("ties_at_thresh", ctypes.c_int64),
                ("ties_taken", ctypes.c_int64)]


class IsoMergeStats(ctypes.Structure):
    _fields_ = [("status", ctypes.c_void_p), ("units", ctypes.c_void_p),
                ("gram", ctypes.c_void_p), ("coef", ctypes.c_void_p)]


class IsoFrameCfg(ctypes.Structure):
    _fields_ = [("rho_keep", ctypes.c_double), ("ridge", ctypes.c_double), ("c_min", ctypes.c_double),
                ("c_max", ctypes.c_double), ("ns_iters", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class IsoAdamwCfg(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_double), ("beta1", ctypes.c_double), ("beta2", ctypes.c_double),
                ("eps", ctypes.c_double), ("weight_decay", ctypes.c_double), ("step", ctypes.c_int64),
                ("ns_iters", ctypes.c_int32), ("reserved", ctypes.c_int32)]


# (name, restype, argtypes) for every entry point of include/iso.h
P = ctypes.c_void_p
PT = ctypes.POINTER(IsoTensor)
I32, I64, SZ = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
PROTOTYPES = [
    ("iso_num_units", I32, [PT, I32, ctypes.POINTER(IsoTopkCfg), ctypes.POINTER(I64)]),
    ("iso_workspace_size", I32, [PT, I32, I32, ctypes.POINTER(IsoMergeCfg), ctypes.POINTER(SZ),
                                 ctypes.POINTER(SZ)]),
    ("iso_delta", I32, [PT, PT, PT, I32, P]),
    ("iso_topk_mask", I32, [PT, I32, ctypes.POINTER(IsoTopkCfg), P, ctypes.POINTER(IsoMergeStats),
                            P, SZ, P]),
    ("iso_update", I32, [PT, PT, I32, PT, I32, ctypes.POINTER(IsoMergeCfg), P, SZ,
                         ctypes.POINTER(IsoMergeStats), P]),
    ("iso_merge", I32, [PT, PT, I32, I32, PT, I32, ctypes.POINTER(IsoMergeCfg), P, SZ,
                        ctypes.POINTER(IsoMergeStats), P]),
    ("iso_update_noalloc", I32, [PT, PT, I32, PT, I32, ctypes.POINTER(IsoMergeCfg),
                                 ctypes.POINTER(IsoMergeStats), P]),
    ("iso_range_hist", I32, [PT, PT, I64, I64, ctypes.c_uint32, I32, I32, I32, P, P]),
    ("iso_range_mask_workspace_size", I32, [I64, ctypes.POINTER(SZ)]),
    ("iso_range_mask", I32, [PT, PT, I64, I64, ctypes.c_uint32, I64, P, P, SZ, P]),
    ("iso_update_host_staging_size", I32, [PT, PT, PT, I32, ctypes.POINTER(IsoMergeCfg), SZ,
                                           ctypes.POINTER(SZ)]),
    ("iso_update_host", I32, [PT, PT, I32, PT, I32, ctypes.POINTER(IsoMergeCfg), SZ, P, SZ,
                              ctypes.POINTER(IsoMergeStats), ctypes.POINTER(P)]),
    ("iso_frame_workspace_size", I32, [I64, I64, I32, ctypes.POINTER(SZ)]),
    ("iso_frame_merge", I32, [P, P, P, P, P, I32, I64, I64, PT, PT, ctypes.POINTER(IsoFrameCfg), P, SZ,
                              ctypes.POINTER(IsoMergeStats), P]),
    ("iso_gemm_tf32", I32, [P, I64, P, I64, P, I64, I64, I64, I64, I64, I64, P]),
    ("iso_opt_workspace_size", I32, [I64, I64, ctypes.POINTER(SZ)]),
    ("iso_opt_step", I32, [P, P, P, PT, P, P, P, P, PT, PT, I64, I64, ctypes.POINTER(IsoAdamwCfg), P, SZ,
                           ctypes.POINTER(IsoMergeStats), P]),
    ("iso_error_string", ctypes.c_char_p, [I32]),
    ("iso_launch_count", ctypes.c_uint64, []),
    ("iso_force_two_pass", ctypes.c_int32, [ctypes.c_int32]),
    ("iso_compact_candidates", ctypes.c_int32, [ctypes.c_int32]),
    ("iso_profile_enable", I32, [I32]),
    ("iso_profile_reset", I32, []),
    ("iso_profile_kinds", I32, []),
    ("iso_profile_name", ctypes.c_char_p, [I32]),
    ("iso_profile_read", I32, [I32, ctypes.POINTER(I64), ctypes.POINTER(ctypes.c_double)]),
]

_lock = threading.Lock()
_lib = None


class IsoError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        msg = lib().iso_error_string(code).decode() if _lib is not None else str(code)
        super().__init__(f"{where}: {msg} ({code})")


def lib():
    """The loaded library; raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(
                    f"libiso_gb300.so not found at {LIB_PATH}: build it first "
                    "(python -c 'import __graft_entry__ as g; g.build()')")
            h = ctypes.CDLL(LIB_PATH)
            for name, res, args in PROTOTYPES:
                fn = getattr(h, name)
                fn.restype = res
                fn.argtypes = args
            _lib = h
    return _lib


def check(code: int, where: str) -> None:
    if code != ISO_OK:
        raise IsoError(code, where)
