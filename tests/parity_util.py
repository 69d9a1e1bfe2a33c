"""Comparison helpers for the GPU-vs-oracle parity tests.

Tolerances.  The oracle computes values in binary64 and rounds once to the
output encoding; the kernels compute in binary32 with one rounding per
operation, the experts summed in a fixed order.

* binary32 outputs: |gpu - oracle| <= 1e-6 |oracle| (the bound the workload
  specification states), except where the update cancels against theta_0 or
  the experts cancel among themselves.  There the binary32 error is bounded
  by r 2^-24 M, with M = |theta_0| + the sum of the magnitudes of the
  update's terms at that entry and r the number of binary32 roundings on the
  path (``rounding_steps``), and that bound is used instead.
* bfloat16 outputs: |gpu - oracle| <= 1 bfloat16 ulp: both sides round once
  to bfloat16, so they agree or are neighbours.  The cancellation bound
  above replaces the ulp only where it is the larger one, i.e. where the
  output is below about 2^-16 r M.

Each check records its worst observed error (relative error for binary32,
ulps for bfloat16) and how many entries needed the cancellation bound; the
session prints the table at the end (tests/conftest.py), so the slack each
test leaves is visible in its output.
"""
import numpy as np
import torch

U32 = 2.0 ** -24
# what -> (worst relative error or ulps, entries checked, entries on the cancellation bound, kind)
WORST = {}


def rounding_steps(op: str = "iso", K: int = 8) -> int:
    """binary32 roundings between the exact inputs and the unrounded output.

    TA:   K - 1 adds, the scale, the add to theta_0            -> K + 1
    TIES: K - 1 adds, the division, the scale, the add          -> K + 2
    RAM:  as TIES                                               -> K + 2
    ISO:  K products c_i tau_i, K adds (theta_0 first), and the
          binary32 coefficient itself (c* is solved in binary64
          from a Gram summed in another order than the oracle's) -> 2K + 2
    The checkpoint difference tau = x - theta_0 is one more rounding.
    """
    base = {"ta": K + 1, "ties": K + 2, "ram": K + 2, "iso": 2 * K + 2}[op]
    return base + 1


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


def _record(what: str, worst: float, n: int, n_cancel: int, kind: str):
    key = what.split(" tensor ")[0]
    w0, n0, c0, _ = WORST.get(key, (0.0, 0, 0, kind))
    WORST[key] = (max(w0, worst), n0 + n, c0 + n_cancel, kind)


def assert_values_close(gpu: np.ndarray, out64: np.ndarray, mag: np.ndarray, what="",
                        op: str = "iso", K: int = 8):
    """gpu: uint16 (bfloat16 bits) or float32 array; out64/mag: binary64."""
    r = rounding_steps(op, K)
    cancel = r * U32 * mag
    if gpu.dtype == np.uint16:
        g = bf16_value(gpu)
        ulp = bf16_ulp(np.maximum(np.abs(g), np.abs(out64)))
        plain = ulp
        kind = "ulp"
    else:
        g = gpu.astype(np.float64)
        plain = 1e-6 * np.abs(out64)
        ulp = None
        kind = "rel"
    err = np.abs(g - out64)
    tol = np.maximum(plain, cancel)
    bad = err > tol
    if bad.any():
        i = np.flatnonzero(bad)[:5]
        raise AssertionError(f"{what}: {bad.sum()} / {bad.size} entries outside tolerance; "
                             f"first {i.tolist()}: gpu {g[i].tolist()} oracle {out64[i].tolist()} "
                             f"tol {tol[i].tolist()}")
    n_cancel = int(np.count_nonzero(err > plain))
    if err.size:
        if kind == "ulp":
            worst = float(np.max(err / ulp))
        else:
            nz = out64 != 0
            worst = float(np.max(err[nz] / np.abs(out64[nz]))) if nz.any() else 0.0
        _record(what, worst, int(err.size), n_cancel, kind)


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
