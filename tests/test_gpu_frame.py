"""GPU parity of the frame-space ISO-Merger (App. E) and of its tensor-core
product, through the C ABI.

* iso_gemm_tf32 (tcgen05.mma, operands staged by TMA, accumulator in tensor
  memory): on operands whose products and sums are exact in binary32 (small
  multiples of 1/8) the result must equal the binary64 product bit for bit,
  over several output tiles, a ring of stages that wraps many times and
  contraction offsets.
* iso_frame_merge against oracle/iso_merger.py on tall, wide and square
  matrices, K = 1 ... 8 experts, rho_keep 0.5 / 0.9 / 1, binary32 and
  bfloat16 weights.  The GPU is given the oracle's own thin-SVD factors, so
  the comparison isolates the merge.  Tolerances are derived from the
  arithmetic: every large contraction is three tf32 products per pair
  (about 2^-22 relative each) accumulated in binary32 over N = 3 max(m, n)
  terms, so a computed quantity is accurate to eps = 4 * 2^-24 (8 + sqrt N)
  of the magnitude of its terms before they cancel:
    Gamma_ij   |err| <= eps (a_i + b_i)(a_j + b_j), a_i = ||xi~_Ui S_0||_F,
               b_i = ||xi~_Vi S_0||_F (the two halves of the proxy g_i);
    c*         the solve's first-order bound 2 ||(Gamma + ridge I)^-1||_2
               ||dGamma||_F (1 + ||c*||_2) over the active experts;
    W*         |err| <= eps (|E_U| |S_0| |V*|^T + |U_0| |S_0| |E_V|^T)
               + sum_i |dc_i| |g_i| + one rounding of the output, E_F = F* - F_0;
               for bfloat16 outputs one ulp of the oracle's value unless
               that bound is larger.
  Near-degenerate spectra (the test bases' consecutive singular values are
  closer than the experts' perturbations) make the frames rotate far while
  the proxies stay small, so these bounds are far above |Gamma| and |W* -
  W_0| there; the worst observed error against each bound is reported.
  The spectrum of W* equals the base's within the same bound (Weyl's
  inequality) and experts equal to the base leave W_0 bit for bit.
"""
import numpy as np
import pytest
import torch

import paper_2607_19331_gb300 as iso
from oracle import iso_merger as M
from paper_2607_19331_gb300 import _abi
from parity_util import bf16_ulp

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()


# ---------------------------------------------------------------------------
# the tensor-core product
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("M_,N_,Kc,a_k0,b_k0,lda,ldb", [
    (128, 128, 32, 0, 0, 32, 32),            # one tile, one stage
    (256, 384, 1024, 0, 64, 1024, 1088),     # 6 tiles, the six-stage ring wraps five times
    (384, 128, 224, 32, 0, 256, 224),        # offsets, a contraction of seven stages
    (128, 256, 3072, 1024, 0, 4096, 3072),   # the split layout's segment offsets
])
def test_gemm_tf32_exact(M_, N_, Kc, a_k0, b_k0, lda, ldb):
    g = torch.Generator().manual_seed(M_ * 7 + Kc)
    A = (torch.randint(-8, 9, (M_, lda), generator=g).float() / 8).to(DEV)
    B = (torch.randint(-8, 9, (N_, ldb), generator=g).float() / 8).to(DEV)
    C = torch.full((M_, N_), float("nan"), device=DEV)
    iso.gemm_tf32(A, B, C, Kc, a_k0, b_k0)
    torch.cuda.synchronize()
    ref = A[:, a_k0:a_k0 + Kc].double() @ B[:, b_k0:b_k0 + Kc].double().T
    assert torch.equal(C.double(), ref), float((C.double() - ref).abs().max())


def test_gemm_tf32_rounding_of_general_operands():
    # general binary32 operands are read as tf32 (10 mantissa bits): the error
    # stays within the tf32 bound of the product's magnitude
    g = torch.Generator().manual_seed(5)
    A = torch.randn(256, 512, generator=g).to(DEV)
    B = torch.randn(128, 512, generator=g).to(DEV)
    C = torch.empty(256, 128, device=DEV)
    iso.gemm_tf32(A, B, C, 512)
    torch.cuda.synchronize()
    ref = A.double() @ B.double().T
    mag = A.double().abs() @ B.double().abs().T
    assert ((C.double() - ref).abs() <= 2.0 ** -10 * mag).all()


# ---------------------------------------------------------------------------
# the frame-space merge
# ---------------------------------------------------------------------------
def _orth(rng, m, q):
    Q, R = np.linalg.qr(rng.normal(size=(m, q)))
    return Q * np.sign(np.diag(R))


def _case(seed, m, n, K, dtype=np.float32, motion=0.05):
    """A base with evenly spaced singular values and K experts moved by
    `motion` (relative), stored in `dtype` (the oracle sees the stored
    values).  At motion 0.05 the perturbation exceeds the spectral gaps (large
    frame rotations, small proxies); at 0.001 it stays well below them."""
    rng = np.random.default_rng(seed)
    q = min(m, n)
    U, V = _orth(rng, m, q), _orth(rng, n, q)
    S = np.linspace(2.0, 0.2, q) * 0.05
    W0 = (U * S) @ V.T
    ex = [W0 + motion * 0.05 * rng.normal(size=(m, n)) / np.sqrt(max(m, n)) for _ in range(K)]
    if dtype == "bf16":
        cast = lambda a: torch.from_numpy(a).to(torch.bfloat16)
    else:
        cast = lambda a: torch.from_numpy(a.astype(np.float32))
    W0_t, ex_t = cast(W0), [cast(e) for e in ex]
    return W0_t, ex_t, W0_t.double().numpy(), [e.double().numpy() for e in ex_t]


def _factors_on_gpu(W):
    U, S, V = M.thin_svd(W)
    to = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(DEV)
    return to(U), to(S), to(V.T)


def _run(W0_t, W0, experts, **kw):
    U0, S0, Vt0 = _factors_on_gpu(W0)
    Us, Vts = [], []
    for E in experts:
        U, _, Vt = _factors_on_gpu(E)
        Us.append(U)
        Vts.append(Vt)
    out, st = iso.frame_merge_factors(U0, S0, Vt0, Us, Vts, W0_t.to(DEV), stats=True, **kw)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    return out.cpu(), st


def _eps(m, n):
    return 4 * 2.0 ** -24 * (8 + np.sqrt(3 * max(m, n)))


def _check(out, st, r, W0, what):
    """The GPU's Gamma, c* and W* against the oracle's, within the bounds
    derived in the module docstring; returns the worst error / bound ratios."""
    m, n = W0.shape
    eps = _eps(m, n)
    S0 = r["S0"]
    K = r["coef"].size
    gram = st.gram.cpu().numpy()
    coef = st.coef.cpu().numpy()
    a = np.array([np.linalg.norm(x * S0[None, :]) for x in r["xiU"]])
    b = np.array([np.linalg.norm(x * S0[None, :]) for x in r["xiV"]])
    dG = eps * np.outer(a + b, a + b)
    ratio = {"gram": float(np.max(np.abs(gram - r["gram"]) / (dG + 1e-300)))}
    assert ratio["gram"] <= 1.0, (what, gram, r["gram"], dG)
    act = np.flatnonzero(np.diag(r["gram"]) > 0)
    if act.size:
        Ga = r["gram"][np.ix_(act, act)] + 1e-12 * np.eye(act.size)
        dc = 2 * np.linalg.norm(np.linalg.inv(Ga), 2) * np.linalg.norm(dG[np.ix_(act, act)]) * \
            (1 + np.linalg.norm(r["coef"]))
    else:
        dc = 0.0
    dc = max(dc, 1e-12)
    ratio["coef"] = float(np.max(np.abs(coef - r["coef"])) / dc)
    assert ratio["coef"] <= 1.0, (what, coef, r["coef"], dc)
    want = r["W"]
    EU, EV = np.abs(r["U"] - r["U0"]), np.abs(r["V"] - r["V0"])
    sa = np.abs(S0)[None, :]
    bound = eps * ((EU * sa) @ np.abs(r["V"]).T + (np.abs(r["U0"]) * sa) @ EV.T)
    bound += dc * sum(np.abs(g) for g in r["g"])
    if out.dtype == torch.bfloat16:
        got = out.float().double().numpy()
        bound = np.maximum(bound, bf16_ulp(np.maximum(np.abs(got), np.abs(want))))
    else:
        got = out.double().numpy()
        bound = bound + 2.0 ** -23 * np.abs(want)
    err = np.abs(got - want)
    ratio["W"] = float(np.max(err / bound))
    assert ratio["W"] <= 1.0, (what, float(err.max()), ratio)
    # the fixed-spectrum property (Weyl: singular values move by at most the
    # spectral norm of the perturbation, here below the bound's Frobenius norm)
    s0 = np.linalg.svd(W0, compute_uv=False)
    s1 = np.linalg.svd(got, compute_uv=False)
    assert np.abs(s1 - s0).max() <= np.linalg.norm(bound) + 1e-12 * s0.max(), what
    WORST_FRAME[what] = ratio
    return ratio


WORST_FRAME = {}


@pytest.mark.parametrize("m,n,K,rho,motion", [
    (96, 64, 3, 0.9, 0.05),       # tall, one tile
    (64, 160, 2, 0.9, 0.05),      # wide
    (80, 80, 4, 0.9, 0.05),       # square
    (300, 200, 1, 0.9, 0.05),     # one expert, ragged padding
    (200, 520, 8, 0.9, 0.05),     # eight experts, wide, several tiles along n
    (384, 256, 2, 0.5, 0.05),     # half the modes masked, several tiles along q
    (160, 144, 3, 1.0, 0.05),     # no mode masked
    (256, 384, 3, 0.9, 0.001),    # motion well inside the spectral gaps
])
def test_frame_merge_matches_oracle(m, n, K, rho, motion):
    W0_t, ex_t, W0, ex = _case(m * 1000 + n + K, m, n, K, motion=motion)
    r = M.merge_matrix(W0, ex, rho_keep=rho)
    out, st = _run(W0_t, W0, ex, rho_keep=rho)
    _check(out, st, r, W0, f"{m}x{n} K={K} rho={rho}")


def test_frame_merge_bf16_weights():
    W0_t, ex_t, W0, ex = _case(11, 192, 320, 3, dtype="bf16")
    r = M.merge_matrix(W0, ex)
    out, st = _run(W0_t, W0, ex)
    assert out.dtype == torch.bfloat16
    _check(out, st, r, W0, "bf16 192x320")


def test_frame_merge_experts_equal_to_base_is_a_fixed_point():
    W0_t, _, W0, _ = _case(12, 130, 90, 1)
    out, st = _run(W0_t, W0, [W0, W0])
    assert torch.equal(out, W0_t)
    assert (st.coef.cpu().numpy() == 0).all()


def test_frame_merge_in_place_and_through_gpu_svds():
    # the GPU's own thin SVDs (torch.linalg in binary64) instead of the oracle's
    # factors: the singular vectors differ by rounding and by sign, which the
    # sign gauge absorbs; and out may coincide with W0
    W0_t, ex_t, W0, ex = _case(13, 144, 208, 2)
    r = M.merge_matrix(W0, ex)
    W = W0_t.to(DEV)
    out, st = iso.frame_merge(W, [e.to(DEV) for e in ex_t], out=W, stats=True)
    torch.cuda.synchronize()
    assert out.data_ptr() == W.data_ptr()
    _check(out.cpu(), st, r, W0, "torch SVDs, in place")


def test_frame_merge_full_size_projection():
    # one Qwen2.5-7B gate/up projection (3584 x 18944, bf16), two RL experts,
    # through the GPU's own thin SVDs, against the oracle in binary64
    m, n, K = 3584, 18944, 2
    g = torch.Generator().manual_seed(7)
    W0 = (torch.randn(m, n, generator=g) * 0.02).to(torch.bfloat16)
    ex = [(W0.float() + torch.randn(m, n, generator=g) * 5e-4).to(torch.bfloat16) for _ in range(K)]
    W0n = W0.double().numpy()
    r = M.merge_matrix(W0n, [e.double().numpy() for e in ex])
    out, st = iso.frame_merge(W0.to(DEV), [e.to(DEV) for e in ex], stats=True)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    _check(out.cpu(), st, r, W0n, "Qwen2.5-7B gate 3584x18944 K=2 bf16 (GPU SVDs)")
    del out, st
    torch.cuda.empty_cache()
