"""Frame-space ISO-Merger (App. E) -- TEST INFRASTRUCTURE ONLY.

A plain binary64 numpy restatement of the definitions of App. E, one small
function per definition, each citing the subsection that defines it; the
merge of one matrix composes them.  Library routines serve where the paper
names the operation (the thin SVD, matrix products); nothing is blocked,
fused or reordered.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline leg may import it; it shares no code with the
CUDA library.

Definitions (App. E):

* Setup: the shared base and every expert as thin SVDs W = U S V^T with
  q = min(m, n) singular values in descending order; the merged matrix keeps
  the base spectrum S_0 and moves only the frames.
* Sign canonicalization: an SVD fixes each mode (u_k, v_k) only up to a joint
  sign, so each expert mode takes s_k = sign(<u_0k, u_k>), sign(0) := 1, on
  both of its frames.
* Stiefel tangent projection: the tangent space at U_0 is
  {xi : U_0^T xi + xi^T U_0 = 0} and the orthogonal projection onto it is
  Pi_{U_0}(D) = D - U_0 sym(U_0^T D); an expert's frame motion is the
  projected displacement of its aligned frames from the base's.
* Top-k_keep singular-mode masking: D_keep keeps the leading
  k_keep = round(rho_keep q) modes (halves rounded up) of each displacement.
* Retention coefficients: the effect proxy g_i = xi~_Ui S_0 V_0^T +
  U_0 S_0 xi~_Vi^T, its Gram matrix Gamma_ij = <g_i, g_j>_F and the clipped
  solution of (Gamma + ridge I) c = diag Gamma on the non-zero proxies (the
  element-wise oracle's pinned solve).
* Retraction and reconstruction: the aggregate xi_* = Pi_{U_0}(sum_i c_i
  xi~_Ui) (same for V), the polar factor polar(X) = P Q^T of the thin SVD
  X = P S Q^T, U_* = polar(U_0 + xi_U*), and W_* = U_* S_0 V_*^T.
* Merged parameter scope: one-dimensional parameters take the task-vector
  average w_0 + (1/K) sum_i (w_i - w_0); ``merge_model`` applies the matrix
  merge or the average to each tensor of a list and rounds each result once
  to the base's encoding.

Parity status: pinned (tests/test_oracle_iso_merger.py) by the identities the
paper states -- the tangent condition, (U_0 + xi)^T (U_0 + xi) = I + xi^T xi,
polar(X) = X (X^T X)^{-1/2} for full column rank -- and by the spectrum of
W* equal to that of W_0, fixed points (experts equal to the base, zero
coefficients), sign-flip invariance, the mode mask, the single-expert
third-order accuracy of the retraction, identical experts, the Gram and the
aggregate projection in their q x q forms, and the model loop against the
element-wise oracle's 1-D rule.
"""
from __future__ import annotations

import numpy as np

from . import retention as _retention


def sym(A: np.ndarray) -> np.ndarray:
    """sym(A) = (A + A^T) / 2."""
    return 0.5 * (A + A.T)


def tangent_project(U0: np.ndarray, D: np.ndarray) -> np.ndarray:
    """Orthogonal projection onto the tangent space of the Stiefel manifold
    at U0: Pi_{U0}(D) = D - U0 sym(U0^T D)."""
    return D - U0 @ sym(U0.T @ D)


def thin_svd(W: np.ndarray):
    """W = U diag(S) V^T with q = min(m, n) singular values, descending."""
    U, S, Vt = np.linalg.svd(np.asarray(W, np.float64), full_matrices=False)
    return U, S, Vt.T


def canonicalize_signs(U0: np.ndarray, U: np.ndarray, V: np.ndarray):
    """Joint per-mode sign alignment of (U, V) against the base frame U0:
    s_k = sign(<u0_k, u_k>), sign(0) := 1; both frames take the same sign,
    which leaves U diag(S) V^T unchanged."""
    s = np.sign(np.sum(U0 * U, axis=0))
    s[s == 0] = 1.0
    return U * s, V * s, s


def k_keep_of(rho_keep: float, q: int) -> int:
    """k_keep = round(rho_keep q), rounding halves up (floor(x + 1/2)),
    clamped to [0, q]."""
    k = int(np.floor(rho_keep * q + 0.5))
    return max(0, min(q, k))


def keep_mask(xi: np.ndarray, k_keep: int) -> np.ndarray:
    """xi D_keep: the leading k_keep columns kept, the trailing ones zeroed."""
    out = xi.copy()
    out[:, k_keep:] = 0.0
    return out


def effect_proxy(xiU: np.ndarray, xiV: np.ndarray, U0: np.ndarray, S0: np.ndarray,
                 V0: np.ndarray) -> np.ndarray:
    """g = xi_U S_0 V_0^T + U_0 S_0 xi_V^T."""
    return (xiU * S0) @ V0.T + (U0 * S0) @ xiV.T


def polar(X: np.ndarray) -> np.ndarray:
    """polar(X) = P Q^T from the thin SVD X = P S Q^T."""
    P, _, Q = thin_svd(X)
    return P @ Q.T


def expert_motion(U0: np.ndarray, V0: np.ndarray, Wi: np.ndarray, k_keep: int):
    """One expert's masked frame motion (App. E, Sign canonicalization,
    Stiefel tangent projection and Top-k_keep masking): its thin-SVD frames
    in the base's sign gauge, their displacements from (U0, V0) projected
    onto the tangent spaces there, the trailing modes zeroed.  Returns
    (xi~_U, xi~_V, signs)."""
    Ui, _, Vi = thin_svd(Wi)
    Ui, Vi, s = canonicalize_signs(U0, Ui, Vi)
    xu = keep_mask(tangent_project(U0, Ui - U0), k_keep)
    xv = keep_mask(tangent_project(V0, Vi - V0), k_keep)
    return xu, xv, s


def gram_matrix(g) -> np.ndarray:
    """Gamma_ij = <g_i, g_j>_F (App. E, Retention coefficients)."""
    K = len(g)
    gram = np.zeros((K, K), np.float64)
    for i in range(K):
        for j in range(K):
            gram[i, j] = float(np.sum(g[i] * g[j]))
    return gram


def aggregate_tangent(U0: np.ndarray, xis, c) -> np.ndarray:
    """xi_* = Pi_{U0}(sum_i c_i xi~_i) (App. E, Retraction and reconstruction)."""
    agg = np.zeros_like(U0)
    for i in range(len(xis)):
        agg += c[i] * xis[i]
    return tangent_project(U0, agg)


def retract(U0: np.ndarray, xi: np.ndarray) -> np.ndarray:
    """The merged frame polar(U0 + xi) (App. E, Retraction and reconstruction)."""
    return polar(U0 + xi)


def merge_matrix(W0, experts, rho_keep=0.9, ridge=1e-12, c_min=0.0, c_max=1.5):
    """ISO-Merger of one 2-D weight matrix (App. E).

    W0       base matrix (m x n)
    experts  list of K expert matrices of the same shape (checkpoints W_i)

    Returns a dict: ``W`` (merged matrix, binary64), ``U``, ``V`` (merged
    frames), ``S0``, ``U0``, ``V0``, ``k_keep``, ``coef`` (c*), ``gram``
    (Gamma), ``g`` (proxies), ``xiU`` / ``xiV`` (masked tangents per expert),
    ``xiU_star`` / ``xiV_star`` (aggregate tangents) and ``signs``.
    """
    W0 = np.asarray(W0, np.float64)
    U0, S0, V0 = thin_svd(W0)
    kk = k_keep_of(rho_keep, S0.size)
    motion = [expert_motion(U0, V0, np.asarray(Wi, np.float64), kk) for Wi in experts]
    xiU = [m[0] for m in motion]
    xiV = [m[1] for m in motion]
    signs = [m[2] for m in motion]
    g = [effect_proxy(xu, xv, U0, S0, V0) for xu, xv in zip(xiU, xiV)]
    gram = gram_matrix(g)
    # zero-norm proxies are dropped inside the solve (coefficient 0)
    coef = _retention(gram, ridge, c_min, c_max)
    xiU_star = aggregate_tangent(U0, xiU, coef)
    xiV_star = aggregate_tangent(V0, xiV, coef)
    U_star = retract(U0, xiU_star)
    V_star = retract(V0, xiV_star)
    W_star = (U_star * S0) @ V_star.T
    return {"W": W_star, "U": U_star, "V": V_star, "S0": S0, "U0": U0, "V0": V0,
            "k_keep": kk, "coef": coef, "gram": gram, "g": g, "xiU": xiU, "xiV": xiV,
            "xiU_star": xiU_star, "xiV_star": xiV_star, "signs": signs}


def merge_model(theta0, experts, is_1d=None, rho_keep=0.9, ridge=1e-12, c_min=0.0, c_max=1.5):
    """The merge of a parameter list (App. E, Merged parameter scope).

    theta0   list of base tensors (uint16 bfloat16 bits or float32), 2-D
             matrices as (m, n) arrays
    experts  K lists of checkpoints in the same encoding
    is_1d    per tensor: 1-D parameters take the task-vector average
             w_0 + (1/K) sum_i (w_i - w_0); every other tensor is merged as a
             matrix with ``merge_matrix``

    Returns the merged tensors in the base encoding (one rounding from
    binary64) and the per-matrix results (None for 1-D tensors)."""
    from . import BF16, F32, load, to_dtype
    K = len(experts)
    if is_1d is None:
        is_1d = [np.asarray(a).ndim == 1 for a in theta0]
    out, detail = [], []
    for t, a in enumerate(theta0):
        a = np.asarray(a)
        code = F32 if a.dtype == np.float32 else BF16
        _, w0 = load(a)
        ws = [load(np.asarray(experts[i][t]))[1] for i in range(K)]
        if is_1d[t]:
            s = np.zeros_like(w0)
            for w in ws:
                s += w - w0
            # an update of exactly zero keeps the base's bits (a -0 stays -0)
            merged = np.where(s == 0.0, w0, w0 + s / K)
            detail.append(None)
        else:
            r = merge_matrix(w0.reshape(a.shape), [w.reshape(a.shape) for w in ws],
                             rho_keep, ridge, c_min, c_max)
            merged = r["W"].reshape(-1)
            detail.append(r)
        out.append(to_dtype(merged, code).reshape(a.shape))
    return out, detail
