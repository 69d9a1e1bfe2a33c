"""Pins of the frame-space ISO-Merger oracle (App. E).

Each test ties the oracle to a fact fixed outside its code: an identity the
paper states (the Stiefel tangent condition, (U_0 + xi)^T (U_0 + xi) =
I + xi^T xi for a tangent xi, polar(X) = X (X^T X)^{-1/2} at full column rank,
W* carrying the base spectrum), a fixed point, the joint sign gauge, the
k_keep rounding, the first-order meaning of the effect proxy, invariance to
the signs an SVD routine picks, and the third-order accuracy of the polar
retraction for a single expert.  All on the CPU, binary64.
"""
import importlib.util
import os

import numpy as np
import pytest


def _load():
    # ISO_MERGER_PATH lets the mutation tests load a deliberately broken copy
    path = os.environ.get("ISO_MERGER_PATH")
    if not path:
        from oracle import iso_merger
        return iso_merger
    spec = importlib.util.spec_from_file_location("iso_merger_mut", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


M = _load()


def _orth(rng, m, q):
    Q, R = np.linalg.qr(rng.normal(size=(m, q)))
    return Q * np.sign(np.diag(R))


def _matrix(rng, m, n, spread=1.0):
    """A generic m x n matrix with well-separated singular values."""
    q = min(m, n)
    U, V = _orth(rng, m, q), _orth(rng, n, q)
    S = np.linspace(2.0, 0.2, q) * spread
    return (U * S) @ V.T, U, S, V


# ---------------------------------------------------------------------------
# building blocks
# ---------------------------------------------------------------------------

def test_tangent_projection():
    rng = np.random.default_rng(0)
    U0 = _orth(rng, 40, 12)
    D = rng.normal(size=(40, 12))
    xi = M.tangent_project(U0, D)
    # tangent condition U0^T xi + xi^T U0 = 0
    np.testing.assert_allclose(U0.T @ xi + xi.T @ U0, 0.0, atol=1e-13)
    # a projection: idempotent, and the identity on tangent vectors
    np.testing.assert_allclose(M.tangent_project(U0, xi), xi, atol=1e-13)
    A = rng.normal(size=(12, 12))
    A = A - A.T
    N = rng.normal(size=(40, 12))
    N = N - U0 @ (U0.T @ N)                       # normal-space part of a tangent vector
    T = U0 @ A + N
    np.testing.assert_allclose(M.tangent_project(U0, T), T, atol=1e-13)
    # and zero on U0 S with S symmetric (the normal space)
    S = rng.normal(size=(12, 12))
    S = S + S.T
    np.testing.assert_allclose(M.tangent_project(U0, U0 @ S), 0.0, atol=1e-12)


def test_retraction_argument_gram_identity():
    rng = np.random.default_rng(1)
    U0 = _orth(rng, 30, 10)
    xi = M.tangent_project(U0, 0.3 * rng.normal(size=(30, 10)))
    X = U0 + xi
    np.testing.assert_allclose(X.T @ X, np.eye(10) + xi.T @ xi, atol=1e-13)


def test_polar_inverse_square_root_form():
    rng = np.random.default_rng(2)
    X = rng.normal(size=(25, 8))
    P = M.polar(X)
    w, E = np.linalg.eigh(X.T @ X)
    want = X @ (E / np.sqrt(w)) @ E.T
    np.testing.assert_allclose(P, want, atol=1e-12)
    np.testing.assert_allclose(P.T @ P, np.eye(8), atol=1e-13)


def test_sign_gauge():
    rng = np.random.default_rng(3)
    W, U, S, V = _matrix(rng, 20, 14)
    flips = np.where(rng.random(14) < 0.5, -1.0, 1.0)
    Uf, Vf = U * flips, V * flips
    np.testing.assert_allclose((Uf * S) @ Vf.T, W, atol=1e-13)     # same matrix
    Ua, Va, s = M.canonicalize_signs(U, Uf, Vf)
    np.testing.assert_array_equal(s, flips)
    np.testing.assert_allclose(Ua, U, atol=1e-15)
    np.testing.assert_allclose(Va, V, atol=1e-15)
    # sign(0) := 1: a mode orthogonal to the base's keeps its sign
    U0 = np.eye(6)[:, :3]
    Ux = np.eye(6)[:, [3, 1, 2]] * np.array([1.0, -1.0, 1.0])
    _, _, s = M.canonicalize_signs(U0, Ux, Ux.copy())
    np.testing.assert_array_equal(s, [1.0, -1.0, 1.0])


@pytest.mark.parametrize("rho,q,want", [(0.9, 10, 9), (0.9, 15, 14), (0.5, 3, 2), (0.25, 2, 1),
                                        (0.9, 1536, 1382), (1.0, 7, 7), (0.0, 7, 0), (0.05, 9, 0)])
def test_k_keep_rounding(rho, q, want):
    # round(rho q) with halves rounded up: 13.5 -> 14, 1.5 -> 2, 0.5 -> 1
    assert M.k_keep_of(rho, q) == want


def test_effect_proxy_is_first_order_change():
    # g = xi_U S0 V0^T + U0 S0 xi_V^T is the first-order change of U S0 V^T
    # when the frames move by the tangents xi_U, xi_V
    rng = np.random.default_rng(4)
    _, U0, S0, V0 = _matrix(rng, 18, 12)
    ZU, ZV = rng.normal(size=U0.shape), rng.normal(size=V0.shape)
    errs = []
    for eps in (1e-3, 5e-4):
        xu = M.tangent_project(U0, eps * ZU)
        xv = M.tangent_project(V0, eps * ZV)
        Ue, Ve = M.polar(U0 + xu), M.polar(V0 + xv)
        change = (Ue * S0) @ Ve.T - (U0 * S0) @ V0.T
        g = M.effect_proxy(xu, xv, U0, S0, V0)
        assert np.linalg.norm(g) > 0.5 * np.linalg.norm(change)
        errs.append(np.linalg.norm(change - g))
    assert 3.0 < errs[0] / errs[1] < 5.0          # the remainder is second order


# ---------------------------------------------------------------------------
# the whole merge of one matrix
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("m,n,K", [(24, 16, 2), (16, 24, 3), (20, 20, 4)])
def test_merged_matrix_keeps_base_spectrum(m, n, K):
    rng = np.random.default_rng(10 + K)
    W0, *_ = _matrix(rng, m, n)
    experts = [W0 + 0.05 * rng.normal(size=(m, n)) for _ in range(K)]
    r = M.merge_matrix(W0, experts)
    s0 = np.linalg.svd(W0, compute_uv=False)
    s = np.linalg.svd(r["W"], compute_uv=False)
    np.testing.assert_allclose(s, s0, rtol=1e-12, atol=1e-13)
    q = min(m, n)
    np.testing.assert_allclose(r["U"].T @ r["U"], np.eye(q), atol=1e-12)
    np.testing.assert_allclose(r["V"].T @ r["V"], np.eye(q), atol=1e-12)
    # the aggregate tangents are tangent at the base frames
    for X0, xi in ((r["U0"], r["xiU_star"]), (r["V0"], r["xiV_star"])):
        np.testing.assert_allclose(X0.T @ xi + xi.T @ X0, 0.0, atol=1e-12)
    # masked modes: the trailing columns of every expert tangent are zero
    kk = r["k_keep"]
    assert kk == int(np.floor(0.9 * q + 0.5))
    for xu, xv in zip(r["xiU"], r["xiV"]):
        assert not xu[:, kk:].any() and not xv[:, kk:].any()
    c = r["coef"]
    assert np.all(c >= 0.0) and np.all(c <= 1.5)


def test_experts_equal_to_base_are_a_fixed_point():
    rng = np.random.default_rng(20)
    W0, *_ = _matrix(rng, 22, 15)
    r = M.merge_matrix(W0, [W0.copy(), W0.copy()])
    np.testing.assert_array_equal(r["coef"], [0.0, 0.0])      # zero proxies are dropped
    np.testing.assert_allclose(r["W"], W0, atol=1e-13)


def test_zero_expert_drops_out():
    rng = np.random.default_rng(21)
    W0, *_ = _matrix(rng, 20, 16)
    E = W0 + 0.05 * rng.normal(size=W0.shape)
    r2 = M.merge_matrix(W0, [E, W0.copy()])
    r1 = M.merge_matrix(W0, [E])
    assert r2["coef"][1] == 0.0
    assert r2["gram"][1, 1] == 0.0 and r2["gram"][0, 1] == 0.0
    np.testing.assert_allclose(r2["coef"][0], r1["coef"][0], rtol=1e-15)
    np.testing.assert_allclose(r2["W"], r1["W"], atol=1e-14)


def test_single_expert_retraction_is_third_order():
    # an expert whose frames moved by eps from the base's with the base
    # spectrum: with every mode kept, W* matches it up to O(eps^3).  The
    # tangent projection of dU = U1 - U0 adds U0 M with M = (dU^T dU) / 2
    # symmetric and O(eps^2) (U1 is orthonormal), and U1 + U0 M =
    # U1 (I + M) + O(eps^3), whose polar factor is U1: the error falls by
    # eight when eps halves
    rng = np.random.default_rng(30)
    W0, U0, S0, V0 = _matrix(rng, 26, 18)
    ZU, ZV = rng.normal(size=U0.shape), rng.normal(size=V0.shape)
    errs, moves = [], []
    for eps in (2e-3, 1e-3):
        U1, V1 = M.polar(U0 + eps * ZU), M.polar(V0 + eps * ZV)
        W1 = (U1 * S0) @ V1.T
        r = M.merge_matrix(W0, [W1], rho_keep=1.0)
        assert r["coef"][0] == pytest.approx(1.0, abs=1e-6)
        errs.append(np.linalg.norm(r["W"] - W1))
        moves.append(np.linalg.norm(W1 - W0))
    assert errs[0] < 1e-3 * moves[0]
    assert 6.0 < errs[0] / errs[1] < 10.0


def test_identical_experts_match_one_expert():
    rng = np.random.default_rng(40)
    W0, *_ = _matrix(rng, 20, 14)
    E = W0 + 0.03 * rng.normal(size=W0.shape)
    r1 = M.merge_matrix(W0, [E])
    for K in (2, 3):
        rk = M.merge_matrix(W0, [E.copy() for _ in range(K)])
        # (G 1 1^T + ridge I) c = G 1: c_i = G / (K G + ridge), sum c = 1 - O(ridge / G)
        assert np.sum(rk["coef"]) == pytest.approx(r1["coef"][0], rel=1e-9)
        np.testing.assert_allclose(rk["W"], r1["W"], atol=1e-9)


def test_trailing_modes_do_not_move_the_merge():
    # an expert that differs from the base only in its trailing (masked)
    # modes contributes nothing: its masked tangents and proxy are zero
    rng = np.random.default_rng(50)
    W0, U0, S0, V0 = _matrix(rng, 24, 20)
    q = S0.size
    kk = M.k_keep_of(0.9, q)
    # rotate the last two modes among themselves: the leading frames stay put
    th = 0.4
    R = np.array([[np.cos(th), -np.sin(th)], [np.sin(th), np.cos(th)]])
    U1, V1 = U0.copy(), V0.copy()
    U1[:, kk:] = U0[:, kk:] @ R
    S1 = S0.copy()
    W1 = (U1 * S1) @ V1.T
    r = M.merge_matrix(W0, [W1])
    # the leading frames agree up to the SVD's rounding: a proxy of ~1e-16
    assert abs(r["coef"][0]) < 1e-9
    assert np.linalg.norm(r["g"][0]) < 1e-12
    np.testing.assert_allclose(r["W"], W0, atol=1e-12)
    # with every mode kept the same expert does move the merge
    r_all = M.merge_matrix(W0, [W1], rho_keep=1.0)
    assert np.linalg.norm(r_all["W"] - W0) > 1e-3


def test_merge_ignores_the_svd_sign_choice(monkeypatch):
    # an SVD routine may return any joint sign per mode; the merge must not
    # depend on it (the gauge canonicalisation of App. E)
    rng = np.random.default_rng(60)
    W0, *_ = _matrix(rng, 21, 17)
    experts = [W0 + 0.04 * rng.normal(size=W0.shape) for _ in range(3)]
    ref = M.merge_matrix(W0, experts)
    real = M.thin_svd
    calls = {"n": 0}

    def flipped(W):
        U, S, V = real(W)
        calls["n"] += 1
        if calls["n"] == 1:
            return U, S, V                     # the base as computed
        f = np.where(np.random.default_rng(calls["n"]).random(S.size) < 0.5, -1.0, 1.0)
        return U * f, S, V * f

    monkeypatch.setattr(M, "thin_svd", flipped)
    got = M.merge_matrix(W0, experts)
    assert calls["n"] >= 4
    np.testing.assert_allclose(got["coef"], ref["coef"], rtol=1e-12)
    np.testing.assert_allclose(got["W"], ref["W"], atol=1e-13)


def test_gram_from_frame_products():
    # <g_i, g_j>_F without the m x n proxies: with P_i = U0^T xi~_Ui and
    # Q_i = V0^T xi~_Vi (U0, V0 orthonormal),
    #   Gamma_ij = sum_k s_k^2 [(xi~_Ui^T xi~_Uj)_kk + (xi~_Vi^T xi~_Vj)_kk]
    #              + tr(S P_i S Q_j) + tr(S P_j S Q_i)
    rng = np.random.default_rng(70)
    for m, n in ((30, 18), (18, 30)):
        W0, *_ = _matrix(rng, m, n)
        experts = [W0 + 0.05 * rng.normal(size=W0.shape) for _ in range(3)]
        r = M.merge_matrix(W0, experts)
        U0, V0, s = r["U0"], r["V0"], r["S0"]
        P = [U0.T @ x for x in r["xiU"]]
        Q = [V0.T @ x for x in r["xiV"]]
        K = len(experts)
        G = np.zeros((K, K))
        for i in range(K):
            for j in range(K):
                d = np.sum(r["xiU"][i] * r["xiU"][j], axis=0) + np.sum(r["xiV"][i] * r["xiV"][j], axis=0)
                G[i, j] = (np.sum(s * s * d) + np.trace((s[:, None] * P[i] * s[None, :]) @ Q[j])
                           + np.trace((s[:, None] * P[j] * s[None, :]) @ Q[i]))
        np.testing.assert_allclose(r["gram"], G, rtol=1e-11, atol=1e-14 * np.abs(G).max())


def test_masked_tangent_base_coordinates_are_skew():
    # U0^T xi_U = skew(U0^T dU) for the projected displacement, so
    # U0^T xi~_U = skew(U0^T dU) D_keep: the aggregate's projection needs only
    # q x q algebra, and the merged frame argument satisfies
    # (U0 + xi*)^T (U0 + xi*) = I + xi*^T xi*
    rng = np.random.default_rng(71)
    W0, *_ = _matrix(rng, 26, 20)
    experts = [W0 + 0.05 * rng.normal(size=W0.shape) for _ in range(2)]
    r = M.merge_matrix(W0, experts)
    U0, kk = r["U0"], r["k_keep"]
    for i, E in enumerate(experts):
        Ui, _, Vi = M.thin_svd(E)
        Ui, Vi, _ = M.canonicalize_signs(U0, Ui, Vi)
        A = U0.T @ (Ui - U0)
        skew = 0.5 * (A - A.T)
        skew[:, kk:] = 0.0
        np.testing.assert_allclose(U0.T @ r["xiU"][i], skew, atol=1e-13)
    agg = sum(c * x for c, x in zip(r["coef"], r["xiU"]))
    B = sum(c * (U0.T @ x) for c, x in zip(r["coef"], r["xiU"]))
    xi_star = agg - U0 @ (0.5 * (B + B.T))
    np.testing.assert_allclose(r["xiU_star"], xi_star, atol=1e-13)
    X = U0 + r["xiU_star"]
    w, Ev = np.linalg.eigh(np.eye(U0.shape[1]) + r["xiU_star"].T @ r["xiU_star"])
    np.testing.assert_allclose(r["U"], X @ (Ev / np.sqrt(w)) @ Ev.T, atol=1e-12)


def test_model_loop_matrices_and_vectors():
    # the parameter-list merge: matrices through the frame-space merge, 1-D
    # parameters through the task-vector average (the element-wise oracle's
    # ISO 1-D rule), each rounded once to the base's encoding
    import oracle
    rng = np.random.default_rng(80)
    W0, *_ = _matrix(rng, 24, 16, spread=0.02)
    b0 = rng.normal(0, 0.02, 16)
    b0[3] = -0.0                                  # kept as -0 where every expert agrees
    theta0 = [oracle.f64_to_bf16(W0), oracle.f64_to_bf16(b0), W0.astype(np.float32)]
    experts = []
    for i in range(3):
        b = b0 + 1e-3 * rng.normal(size=16)
        b[3] = -0.0
        experts.append([oracle.f64_to_bf16(W0 + 1e-3 * rng.normal(size=W0.shape)),
                        oracle.f64_to_bf16(b),
                        (W0 + 1e-3 * rng.normal(size=W0.shape)).astype(np.float32)])
    out, detail = M.merge_model(theta0, experts, is_1d=[False, True, False])
    assert out[0].dtype == np.uint16 and out[1].dtype == np.uint16 and out[2].dtype == np.float32
    assert detail[1] is None
    # the 1-D rule: the element-wise oracle's ISO 1-D average, bit for bit
    r1 = oracle.merge([theta0[1]], [[e[1]] for e in experts], oracle.ISO, experts_are_deltas=False,
                      is_1d=[True])
    np.testing.assert_array_equal(out[1], r1["out"][0])
    assert out[1][3] == 0x8000
    # matrices: the per-matrix merge of the decoded values, rounded once
    for t in (0, 2):
        w0 = oracle.load(theta0[t])[1].reshape(theta0[t].shape)
        ws = [oracle.load(e[t])[1].reshape(theta0[t].shape) for e in experts]
        r = M.merge_matrix(w0, ws)
        np.testing.assert_array_equal(out[t], oracle.to_dtype(r["W"].reshape(-1),
                                                              oracle.F32 if t == 2 else oracle.BF16)
                                      .reshape(theta0[t].shape))
        s = np.linalg.svd(detail[t]["W"], compute_uv=False)
        np.testing.assert_allclose(s, np.linalg.svd(w0, compute_uv=False), rtol=1e-12)
