"""ISO-Optimizer step ISO[AdamW] (Sec. 4.3) -- TEST INFRASTRUCTURE ONLY.

A plain binary64 numpy restatement of one training step of the
fixed-spectrum parameterisation W(U, V) = U S_0 V^T of a 2-D weight, with
AdamW as the base optimizer.  One function per definition; library routines
(matrix products, the thin SVD of the polar factor) serve as steps.  Only
``tests/`` and ``__graft_entry__.smoke()`` may import it; it shares no code
with the CUDA library.

Definitions:
* factor gradients (Sec. 4.3, eq. "iso_factor_gradients"): from the gradient
  G_W with respect to the reconstructed matrix, G_U = G_W V S_0 and
  G_V = G_W^T U S_0 (the chain rule through W = U S_0 V^T);
* the base optimizer on each frame variable with its own state (Sec. 4.3,
  "base optimizer on factors"): AdamW as published (decoupled weight decay,
  Loshchilov and Hutter, ICLR 2019, in the common bias-corrected form):
      m <- b1 m + (1 - b1) g,   v <- b2 v + (1 - b2) g^2,
      X_bar = X - lr wd X - (lr / (1 - b1^t)) m / (sqrt(v / (1 - b2^t)) + eps);
* the feasibility retraction (Sec. 4.3, with the polar factor of App. E):
  U+ = polar(U_bar), V+ = polar(V_bar), polar(X) = P Q^T for the thin SVD
  X = P S Q^T; and W+ = U+ S_0 V+^T, whose singular values are S_0.

Parity status: pinned (tests/test_oracle_iso_optimizer.py) by finite
differences of a quadratic loss through W(U, V) (the factor gradients),
torch.optim.AdamW on the same gradients (the update and its states), the
closed form of a first step (m = g, v = g^2: a step of lr g / (|g| + eps)),
the polar factor's orthonormality and its identity X (X^T X)^{-1/2}, the
fixed point of a zero gradient, and the spectrum of W+.
"""
from __future__ import annotations

import numpy as np


def factor_gradients(G_W: np.ndarray, U: np.ndarray, S0: np.ndarray, V: np.ndarray):
    """(G_U, G_V) = (G_W V S_0, G_W^T U S_0)."""
    G_W = np.asarray(G_W, np.float64)
    return (G_W @ V) * S0[None, :], (G_W.T @ U) * S0[None, :]


def adamw(X: np.ndarray, g: np.ndarray, m: np.ndarray, v: np.ndarray, step: int, lr: float,
          beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.0):
    """One AdamW update of the variable X (step counted from 1).  Returns the
    tentative X_bar and the new moments (m, v)."""
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    bc1 = 1.0 - beta1 ** step
    bc2 = 1.0 - beta2 ** step
    X_bar = X - lr * weight_decay * X - (lr / bc1) * m / (np.sqrt(v / bc2) + eps)
    return X_bar, m, v


def polar(X: np.ndarray) -> np.ndarray:
    """polar(X) = P Q^T from the thin SVD X = P S Q^T."""
    P, _, Qt = np.linalg.svd(np.asarray(X, np.float64), full_matrices=False)
    return P @ Qt


def step(U, V, S0, G_W, state, t, lr, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0):
    """One ISO[AdamW] step.  state = dict(mU, vU, mV, vV) (binary64 arrays);
    returns dict(U, V, W, state, G_U, G_V, U_bar, V_bar)."""
    U = np.asarray(U, np.float64)
    V = np.asarray(V, np.float64)
    S0 = np.asarray(S0, np.float64)
    G_U, G_V = factor_gradients(G_W, U, S0, V)
    U_bar, mU, vU = adamw(U, G_U, state["mU"], state["vU"], t, lr, beta1, beta2, eps, weight_decay)
    V_bar, mV, vV = adamw(V, G_V, state["mV"], state["vV"], t, lr, beta1, beta2, eps, weight_decay)
    U_new, V_new = polar(U_bar), polar(V_bar)
    W_new = (U_new * S0[None, :]) @ V_new.T
    return {"U": U_new, "V": V_new, "W": W_new, "G_U": G_U, "G_V": G_V, "U_bar": U_bar, "V_bar": V_bar,
            "state": {"mU": mU, "vU": vU, "mV": mV, "vV": vV}}
