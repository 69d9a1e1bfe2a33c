"""Pins of the ISO-Optimizer oracle (Sec. 4.3): each test ties oracle/
iso_optimizer.py to a fact fixed outside its code -- finite differences of a
loss through W(U, V) = U S_0 V^T, PyTorch's own AdamW, the closed form of a
first Adam step, the polar factor's defining properties, a fixed point and
the fixed spectrum.  CPU, binary64."""
import importlib.util
import os

import numpy as np
import pytest
import torch


def _load():
    path = os.environ.get("ISO_OPTIMIZER_PATH")
    if not path:
        from oracle import iso_optimizer
        return iso_optimizer
    spec = importlib.util.spec_from_file_location("iso_optimizer_mut", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


O = _load()


def _orth(rng, m, q):
    Q, R = np.linalg.qr(rng.normal(size=(m, q)))
    return Q * np.sign(np.diag(R))


def _frames(seed, m, n):
    rng = np.random.default_rng(seed)
    q = min(m, n)
    return rng, _orth(rng, m, q), np.linspace(2.0, 0.5, q), _orth(rng, n, q)


def test_factor_gradients_match_finite_differences():
    # L(W) = 1/2 ||W - T||^2 has G_W = W - T; <G_U, D> is the derivative of
    # L(U S V^T) along U + h D (and likewise for V)
    rng, U, S, V = _frames(1, 12, 9)
    T = rng.normal(size=(12, 9))
    loss = lambda U_, V_: 0.5 * np.sum(((U_ * S) @ V_.T - T) ** 2)
    G_W = (U * S) @ V.T - T
    G_U, G_V = O.factor_gradients(G_W, U, S, V)
    h = 1e-6
    for _ in range(3):
        DU, DV = rng.normal(size=U.shape), rng.normal(size=V.shape)
        fd_u = (loss(U + h * DU, V) - loss(U - h * DU, V)) / (2 * h)
        fd_v = (loss(U, V + h * DV) - loss(U, V - h * DV)) / (2 * h)
        assert abs(fd_u - np.sum(G_U * DU)) <= 1e-7 * max(1.0, abs(fd_u))
        assert abs(fd_v - np.sum(G_V * DV)) <= 1e-7 * max(1.0, abs(fd_v))


@pytest.mark.parametrize("wd", [0.0, 0.01])
def test_adamw_matches_torch(wd):
    # three steps of the oracle's AdamW against torch.optim.AdamW on the same
    # gradients (binary64 on the CPU; torch forms the moments by lerp, so the
    # two differ by rounding order: a few ulps)
    rng = np.random.default_rng(2)
    X0 = rng.normal(size=(7, 5))
    grads = [rng.normal(size=(7, 5)) * 10 ** (-k) for k in range(3)]
    p = torch.nn.Parameter(torch.tensor(X0, dtype=torch.float64))
    opt = torch.optim.AdamW([p], lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=wd)
    X, m, v = X0.copy(), np.zeros_like(X0), np.zeros_like(X0)
    for t, g in enumerate(grads, start=1):
        p.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        X, m, v = O.adamw(X, g, m, v, t, 1e-3, 0.9, 0.999, 1e-8, wd)
        np.testing.assert_allclose(X, p.detach().numpy(), rtol=1e-14, atol=1e-17)
        st = opt.state[p]
        np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-14, atol=0)
        np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-14, atol=0)


def test_adamw_first_step_closed_form():
    # t = 1 from zero moments: m^ = g, v^ = g^2, so the step is lr g / (|g| + eps)
    g = np.array([[3.0, -2e-9, 0.0, 1e-3]])
    X, m, v = O.adamw(np.zeros_like(g), g, np.zeros_like(g), np.zeros_like(g), 1, 0.5, 0.9, 0.999, 1e-8, 0.0)
    np.testing.assert_allclose(X, -0.5 * g / (np.abs(g) + 1e-8), rtol=1e-12, atol=0)
    np.testing.assert_allclose(m, 0.1 * g)
    np.testing.assert_allclose(v, 0.001 * g * g)


def test_polar_properties():
    rng = np.random.default_rng(3)
    X = rng.normal(size=(15, 6))
    P = O.polar(X)
    np.testing.assert_allclose(P.T @ P, np.eye(6), atol=1e-13)
    w, E = np.linalg.eigh(X.T @ X)
    np.testing.assert_allclose(P, X @ (E / np.sqrt(w)) @ E.T, atol=1e-12)
    U = _orth(rng, 15, 6)
    np.testing.assert_allclose(O.polar(U), U, atol=1e-13)        # orthonormal frames are fixed


def test_step_keeps_the_spectrum_and_zero_gradient_is_a_fixed_point():
    rng, U, S, V = _frames(4, 20, 14)
    st = {k: np.zeros_like(U if k.endswith("U") else V) for k in ("mU", "vU", "mV", "vV")}
    G_W = rng.normal(size=(20, 14)) * 1e-2
    r = O.step(U, V, S, G_W, st, 1, lr=1e-2)
    np.testing.assert_allclose(np.linalg.svd(r["W"], compute_uv=False), S, rtol=1e-12)
    np.testing.assert_allclose(r["U"].T @ r["U"], np.eye(14), atol=1e-13)
    np.testing.assert_allclose(r["V"].T @ r["V"], np.eye(14), atol=1e-13)
    # to first order the retraction keeps the step's tangent part and drops
    # its normal part: polar(U + D) = U + D - U sym(U^T D) + O(|D|^2)
    D = r["U_bar"] - U
    tang = D - U @ (0.5 * (U.T @ D + D.T @ U))
    assert np.abs(r["U"] - (U + tang)).max() < 4 * np.linalg.norm(D, 2) ** 2
    z = O.step(U, V, S, np.zeros((20, 14)), st, 1, lr=1e-2)
    np.testing.assert_allclose(z["U"], U, atol=1e-14)
    np.testing.assert_allclose(z["W"], (U * S) @ V.T, atol=1e-14)
