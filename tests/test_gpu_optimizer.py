"""GPU parity of the ISO-Optimizer step ISO[AdamW] (Sec. 4.3) through the C
ABI, against oracle/iso_optimizer.py in binary64.

The GPU takes the factor gradients on the tensor cores (three tf32 products
per pair, binary32 accumulation over N = 3 x the contraction) with AdamW in
the products' epilogue (binary64 arithmetic, binary32 moments), then the
polar retraction in difference form and the reconstruction
W+ = W + (U+ S0 V+^T - U S0 V^T).  Bounds, derived from that arithmetic:
* the factor gradient (recovered from the first moment, g = (m+ - b1 m) /
  (1 - b1)) within eps_N (|G_W| |V| S0) plus the moment's binary32 rounding,
  eps_N = 4 * 2^-24 (8 + sqrt N);
* the second moment within (1 - b2)(2 |g| dg + dg^2) plus its rounding;
* the frames: ||U+ - U+_oracle||_F within 1.5 ||d step||_F plus the
  retraction's products, where d step is the AdamW step's change over the
  gradient interval g +- dg (evaluated with the oracle's AdamW);
  |U+^T U+ - I| within 2 |U_bar|^T (eps |U_bar| |R|), R = (U_bar^T
  U_bar)^(-1/2) - I: the retraction's argument U_bar^T U_bar is binary64 and
  only the product U_bar R is tf32 x 3 (the departure is of the order of the
  step times 1e-6 and does not accumulate over steps: each retraction is
  built from the exact U_bar^T U_bar);
* W+ within one bf16 ulp of the oracle's value (bf16 weights), or the change
  the frames' own differences and the products' rounding explain (fp32).
"""
import numpy as np
import pytest
import torch

import paper_2607_19331_gb300 as iso
from oracle import iso_optimizer as O
from paper_2607_19331_gb300 import _abi
from parity_util import bf16_ulp

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
U32 = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()


def _orth(rng, m, q):
    Q, R = np.linalg.qr(rng.normal(size=(m, q)))
    return Q * np.sign(np.diag(R))


def _f32(a):
    return np.asarray(a, np.float32).astype(np.float64)


def _setup(seed, m, n, t, wdtype, gscale=1e-2):
    rng = np.random.default_rng(seed)
    q = min(m, n)
    U, V = _orth(rng, m, q), _orth(rng, n, q)
    S = np.linspace(2.0, 0.5, q) * 0.05
    W = (U * S) @ V.T
    G = _f32(rng.normal(size=(m, n)) * gscale)
    if t == 1:
        st = {k: np.zeros((m if k.endswith("U") else n, q)) for k in ("mU", "vU", "mV", "vV")}
    else:
        st = {}
        for k in ("U", "V"):
            d = m if k == "U" else n
            st["m" + k] = _f32(rng.normal(size=(d, q)) * 1e-3)
            st["v" + k] = _f32(rng.uniform(1e-7, 1e-5, size=(d, q)))
    if wdtype == "bf16":
        W_t = torch.from_numpy(W).to(torch.bfloat16)
    else:
        W_t = torch.from_numpy(W.astype(np.float32))
    return U, V, S, G, st, W_t


def _eps(N):
    return 4 * U32 * (8 + np.sqrt(3 * N))


def _step_interval(g, m_old, v_old, t, lr, b1, b2, eps, wd, X, dg):
    """The AdamW step's largest change over g +- dg (the oracle's own update)."""
    base, _, _ = O.adamw(X, g, m_old, v_old, t, lr, b1, b2, eps, wd)
    dev = np.zeros_like(g)
    for s in (-1.0, -0.5, 0.5, 1.0):
        alt, _, _ = O.adamw(X, g + s * dg, m_old, v_old, t, lr, b1, b2, eps, wd)
        dev = np.maximum(dev, np.abs(alt - base))
    return dev


WORST_OPT = {}


def _run_and_check(m, n, t, wd, wdtype, lr=1e-3, b1=0.9, b2=0.999, eps=1e-8, gscale=1e-2, seed=None):
    U, V, S, G, st, W_t = _setup(seed if seed is not None else m * 10 + n + t, m, n, t, wdtype, gscale)
    r = O.step(U, V, S, G, st, t, lr, b1, b2, eps, wd)
    to = lambda a, dt=torch.float64: torch.from_numpy(np.ascontiguousarray(a)).to(dt).to(DEV)
    Ug, Vg, Sg = to(U), to(V), to(S)
    mom = {k: to(v, torch.float32) for k, v in st.items()}
    out, status = iso.opt_step(Ug, Vg, Sg, to(G, torch.float32), mom["mU"], mom["vU"], mom["mV"], mom["vV"],
                               W_t.to(DEV), lr=lr, beta1=b1, beta2=b2, eps=eps, weight_decay=wd, step=t,
                               stats=True)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    what = f"{m}x{n} t={t} wd={wd} {wdtype}"
    ratio = {}
    q = min(m, n)
    Gabs = np.abs(G)
    for side, F0, Fother, contr in (("U", U, V, n), ("V", V, U, m)):
        mag = (Gabs @ np.abs(Fother) if side == "U" else Gabs.T @ np.abs(Fother)) * S[None, :]
        dg = _eps(contr) * mag
        m_new = mom["m" + side].cpu().double().numpy()
        v_new = mom["v" + side].cpu().double().numpy()
        g_orc = r["G_" + side]
        g_gpu = (m_new - b1 * st["m" + side]) / (1 - b1)
        tol_g = dg + 2 * U32 * (np.abs(m_new) + b1 * np.abs(st["m" + side])) / (1 - b1)
        ratio["g" + side] = float(np.max(np.abs(g_gpu - g_orc) / tol_g))
        assert ratio["g" + side] <= 1.0, (what, side, ratio)
        v_orc = r["state"]["v" + side]
        tol_v = (1 - b2) * (2 * np.abs(g_orc) * tol_g + tol_g ** 2) + 2 * U32 * np.abs(v_orc) + 1e-300
        ratio["v" + side] = float(np.max(np.abs(v_new - v_orc) / tol_v))
        assert ratio["v" + side] <= 1.0, (what, side, ratio)
        d_step = _step_interval(g_orc, st["m" + side], st["v" + side], t, lr, b1, b2, eps, wd, F0, tol_g)
        F_gpu = (Ug if side == "U" else Vg).cpu().numpy()
        dF = r[side + "_bar"] - F0
        tol_F = 1.5 * np.linalg.norm(d_step) + 8 * _eps(2 * max(m, n)) * np.linalg.norm(dF) + 1e-13
        ratio[side] = float(np.linalg.norm(F_gpu - r[side]) / tol_F)
        assert ratio[side] <= 1.0, (what, side, ratio)
        # orthonormality: the retraction's argument is binary64, its product
        # P = F_bar R is tf32 x 3, so F+^T F+ - I is bounded by
        # 2 |F_bar|^T (eps |F_bar| |R|) with R = (F_bar^T F_bar)^(-1/2) - I
        Fb = r[side + "_bar"]
        w, E = np.linalg.eigh(Fb.T @ Fb)
        R = (E / np.sqrt(w)) @ E.T - np.eye(q)
        ortho_bound = 2 * np.abs(Fb).T @ (_eps(q) * (np.abs(Fb) @ np.abs(R))) + 1e-13
        ortho = np.abs(F_gpu.T @ F_gpu - np.eye(q))
        ratio["ortho" + side] = float(np.max(ortho / ortho_bound))
        assert ratio["ortho" + side] <= 1.0, (what, side, ratio)
        ratio["ortho" + side + "_abs"] = float(ortho.max())
    # weights: the oracle's W+ shifted by the stored W's own rounding
    W_store = W_t.double().numpy()
    want = r["W"] + (W_store - (U * S) @ V.T)
    U_g, V_g = Ug.cpu().numpy(), Vg.cpu().numpy()
    dUp, dVp = np.abs(U_g - r["U"]), np.abs(V_g - r["V"])
    EU, EV = np.abs(r["U"] - U), np.abs(r["V"] - V)
    bound = (dUp * S) @ np.abs(r["V"]).T + (np.abs(r["U"]) * S) @ dVp.T \
        + _eps(2 * q) * ((EU * S) @ np.abs(r["V"]).T + (np.abs(U) * S) @ EV.T)
    if wdtype == "bf16":
        got = out.float().double().cpu().numpy()
        bound = np.maximum(bound, bf16_ulp(np.maximum(np.abs(got), np.abs(want))))
    else:
        got = out.double().cpu().numpy()
        bound = bound + 2 * U32 * np.abs(want)
    ratio["W"] = float(np.max(np.abs(got - want) / bound))
    assert ratio["W"] <= 1.0, (what, ratio)
    # the fixed spectrum of the new frames' weights, to first order in their
    # departure from orthonormality
    s_new = np.linalg.svd((U_g * S) @ V_g.T, compute_uv=False)
    dev = np.linalg.norm(U_g.T @ U_g - np.eye(q), 2) + np.linalg.norm(V_g.T @ V_g - np.eye(q), 2)
    np.testing.assert_allclose(s_new, S, rtol=0, atol=2 * dev * S.max() + 1e-13)
    WORST_OPT[what] = ratio


@pytest.mark.parametrize("m,n,t,wd,wdtype", [
    (96, 64, 1, 0.0, "f32"),
    (64, 160, 1, 0.0, "bf16"),
    (300, 200, 5, 0.0, "f32"),
    (256, 384, 5, 0.01, "bf16"),
    (200, 520, 3, 0.0, "f32"),
])
def test_opt_step_matches_oracle(m, n, t, wd, wdtype):
    _run_and_check(m, n, t, wd, wdtype)


def test_opt_step_zero_gradient_is_a_fixed_point():
    U, V, S, _, st, W_t = _setup(21, 130, 90, 1, "f32")
    to = lambda a, dt=torch.float64: torch.from_numpy(np.ascontiguousarray(a)).to(dt).to(DEV)
    Ug, Vg = to(U), to(V)
    mom = {k: to(v, torch.float32) for k, v in st.items()}
    Wg = W_t.to(DEV)
    out = iso.opt_step(Ug, Vg, to(S), torch.zeros(130, 90, device=DEV), mom["mU"], mom["vU"], mom["mV"],
                       mom["vV"], Wg, lr=1e-3, step=1)
    torch.cuda.synchronize()
    assert torch.equal(Ug.cpu(), torch.from_numpy(U)) and torch.equal(Vg.cpu(), torch.from_numpy(V))
    assert torch.equal(out.cpu(), W_t)


def test_opt_step_full_size_projection_paper_learning_rate():
    # one Qwen2.5-7B gate projection (3584 x 18944, bf16 weights) at the
    # paper's ISO-AdamW learning rate 7.5e-7, first step
    _run_and_check(3584, 18944, 1, 0.0, "bf16", lr=7.5e-7, gscale=1e-3, seed=23)
