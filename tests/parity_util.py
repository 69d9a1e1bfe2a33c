"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerances (derived from the arithmetic; the oracle computes values in
binary64, the kernels in binary32 with one rounding per operation and the
experts summed in a fixed order):

* binary32 outputs: |gpu - oracle| <= 1e-6 * M, where M = |theta_0| + the sum
  of the magnitudes of the update's terms at that entry.  With at most K + 2
  binary32 roundings (K <= 8) the error is below (K + 2) 2^-24 M < 1e-6 M.
* bfloat16 outputs: both sides round once to bfloat16; they may differ by one
  bfloat16 ulp at a rounding boundary, plus the binary32 arithmetic error
  1e-6 * M where the output cancels far below its terms.
"""
import numpy as np
import torch


def to_np(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu().contiguous()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16).reshape(-1)
    return t.numpy().reshape(-1)


def bf16_value(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def bf16_ulp(x: np.ndarray) -> np.ndarray:
    a = np.abs(x)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    e = np.maximum(e, -126.0)
    return np.where(a > 0, np.exp2(e - 7.0), np.exp2(-133.0))


def assert_values_close(gpu: np.ndarray, out64: np.ndarray, mag: np.ndarray, what=""):
    """gpu: uint16 (bfloat16 bits) or float32 array; out64/mag: binary64."""
    if gpu.dtype == np.uint16:
        g = bf16_value(gpu)
        tol = np.maximum(bf16_ulp(np.maximum(np.abs(g), np.abs(out64))), 0) + 1e-6 * mag
    else:
        g = gpu.astype(np.float64)
        tol = 1e-6 * mag
    err = np.abs(g - out64)
    bad = err > tol
    if bad.any():
        i = np.flatnonzero(bad)[:5]
        raise AssertionError(f"{what}: {bad.sum()} / {bad.size} entries outside tolerance; "
                             f"first {i.tolist()}: gpu {g[i].tolist()} oracle {out64[i].tolist()} "
                             f"tol {tol[i].tolist()}")


def unpack_mask(words: torch.Tensor, n: int) -> np.ndarray:
    w = words.detach().cpu().numpy().view(np.uint32)
    bits = np.unpackbits(w.view(np.uint8), bitorder="little")
    return bits[:n].astype(np.uint8)


def assert_units_equal(gpu_units: np.ndarray, orc_units: np.ndarray, what=""):
    assert gpu_units.shape == orc_units.shape, (gpu_units.shape, orc_units.shape)
    for f in ("thresh_key", "k", "count_above", "ties_at_thresh", "ties_taken"):
        a, b = gpu_units[f], orc_units[f]
        if not np.array_equal(a, b):
            idx = np.argwhere(a != b)[:5]
            raise AssertionError(f"{what}: unit field {f} differs at {idx.tolist()}: "
                                 f"gpu {[a[tuple(i)] for i in idx]} oracle {[b[tuple(i)] for i in idx]}")
