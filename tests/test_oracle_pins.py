"""Pins of the CPU oracle against facts fixed outside it.

Each test ties the oracle to something other than its own code: a worked
example evaluated by hand in exact rationals, a library sort or linear solve,
a closed form, or an invariant the paper's definitions imply.
"""
import json
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle

HERE = os.path.dirname(os.path.abspath(__file__))


def _golden(name):
    with open(os.path.join(HERE, "golden", name)) as f:
        return json.load(f)


def _fr(v):
    return np.array([float(Fraction(x)) for x in v], np.float64)


def _f32(x):
    return np.asarray(x, np.float32)


# ---------------------------------------------------------------------------
# worked example (App. F TIES / TA, App. E retention, Algorithm 1)
# ---------------------------------------------------------------------------

class TestHandWorked:
    g = _golden("handworked_k2_1x8.json")

    def _inputs(self):
        th0 = _f32(self.g["theta0"]).reshape(1, 8)
        t1 = _f32(_fr(self.g["tau1"])).reshape(1, 8)
        t2 = _f32(_fr(self.g["tau2"])).reshape(1, 8)
        return th0, t1, t2

    @pytest.mark.parametrize("method", ["select", "sort"])
    def test_masks_and_stats(self, method):
        _, t1, t2 = self._inputs()
        k = oracle.k_of(self.g["density"], 8)
        assert k == 4
        for tau, mk, st in ((t1, "mask1", "stats1"), (t2, "mask2", "stats2")):
            m, row = oracle.topk_unit(tau.ravel(), k, method)
            assert m.tolist() == self.g[mk]
            exp = self.g[st]
            assert row["k"] == exp["k"]
            assert row["count_above"] == exp["count_above"]
            assert row["ties_at_thresh"] == exp["ties_at_thresh"]
            assert row["ties_taken"] == exp["ties_taken"]
            assert row["thresh_key"] == np.float32(Fraction(exp["thresh"])).view(np.uint32)

    def test_ties(self):
        th0, t1, t2 = self._inputs()
        r = oracle.merge([th0], [[t1], [t2]], oracle.TIES, density=0.5, lam=1.0, is_1d=[False])
        np.testing.assert_array_equal(r["out64"][0], _fr(self.g["ties"]))
        assert r["out"][0].dtype == np.float32

    def test_ta(self):
        th0, t1, t2 = self._inputs()
        r = oracle.merge([th0], [[t1], [t2]], oracle.TA, lam=1.0, is_1d=[False])
        np.testing.assert_array_equal(r["out64"][0], _fr(self.g["ta"]))

    def test_iso(self):
        th0, t1, t2 = self._inputs()
        r = oracle.merge([th0], [[t1], [t2]], oracle.ISO, density=0.5, is_1d=[False])
        G = np.array([[float(Fraction(x)) for x in row] for row in self.g["iso_gram"]])
        np.testing.assert_array_equal(r["gram"][0], G)
        # the 1e-12 ridge moves c by O(1e-12) relative
        np.testing.assert_allclose(r["coef"][0], _fr(self.g["iso_coef"]), rtol=1e-10)
        np.testing.assert_allclose(r["out64"][0], _fr(self.g["iso"]), rtol=1e-10, atol=1e-12)

    def test_iso_1d_average(self):
        th0, t1, t2 = self._inputs()
        r = oracle.merge([th0.ravel()], [[t1.ravel()], [t2.ravel()]], oracle.ISO,
                         density=0.5, is_1d=[True])
        np.testing.assert_array_equal(r["out64"][0], _fr(self.g["iso_1d"]))


# ---------------------------------------------------------------------------
# TopKMask against a library sort, both oracle methods
# ---------------------------------------------------------------------------

def _sort_reference(tau32, k):
    """Library stable sort on (-key); first k positions."""
    key = (np.asarray(tau32, np.float32).view(np.uint32) & 0x7FFFFFFF).astype(np.int64)
    order = np.argsort(-key, kind="stable")
    m = np.zeros(key.size, np.uint8)
    m[order[:k]] = 1
    return m


def _tie_heavy(rng, n):
    vals = rng.choice(np.array([0.0, 1e-3, -1e-3, 2e-3, -2e-3, 5e-4, 0.25, -0.0], np.float32), n)
    return vals.astype(np.float32)


@pytest.mark.parametrize("seed", range(12))
def test_topk_matches_library_sort(seed):
    rng = np.random.default_rng(seed)
    n = int(rng.integers(1, 4097))
    kind = seed % 3
    if kind == 0:
        tau = rng.normal(0, 1e-3, n).astype(np.float32)
    elif kind == 1:
        tau = _tie_heavy(rng, n)
    else:  # bfloat16-quantised deltas: massive exact ties
        th0 = oracle.f32_to_bf16(rng.normal(0, 0.02, n).astype(np.float32))
        th1 = oracle.f32_to_bf16(oracle.bf16_to_f32(th0) + rng.normal(0, 5e-4, n).astype(np.float32))
        tau, _ = oracle.delta(th1, th0)
    for k in sorted({0, 1, n // 7, n // 2, n - 1, n, int(rng.integers(0, n + 1))}):
        if k < 0:
            continue
        ref = _sort_reference(tau, k)
        for method in ("select", "sort"):
            m, row = oracle.topk_unit(tau, k, method)
            np.testing.assert_array_equal(m, ref, err_msg=f"{method} n={n} k={k}")
            assert int(m.sum()) == k
            assert row["k"] == k


def test_topk_invariants():
    rng = np.random.default_rng(7)
    tau = _tie_heavy(rng, 3001)
    key = tau.view(np.uint32) & 0x7FFFFFFF
    for k in (1, 17, 1500, 3000):
        m, row = oracle.topk_unit(tau, k)
        sel, uns = key[m == 1], key[m == 0]
        assert sel.size == k
        if uns.size:
            assert sel.min() >= uns.max()
        t = row["thresh_key"]
        assert sel.min() == t
        tie_pos = np.nonzero(key == t)[0]
        taken = tie_pos[m[tie_pos] == 1]
        # ties at the threshold: the selected ones are the lowest positions
        assert np.array_equal(taken, tie_pos[:taken.size])
        assert row["count_above"] == int((key > t).sum())
        assert row["ties_at_thresh"] == tie_pos.size
        assert row["ties_taken"] == taken.size


def test_topk_degenerate():
    z = np.zeros(10, np.float32)
    z[3] = -0.0
    m, row = oracle.topk_unit(z, 4)
    assert m.tolist() == [1, 1, 1, 1, 0, 0, 0, 0, 0, 0]   # -0 and +0 tie
    assert row["thresh_key"] == 0 and row["ties_at_thresh"] == 10
    m, row = oracle.topk_unit(z, 0)
    assert m.sum() == 0 and row["thresh_key"] == oracle.KEY_NONE
    m, row = oracle.topk_unit(np.zeros(0, np.float32), 0)
    assert m.size == 0
    m, row = oracle.topk_unit(np.arange(5, dtype=np.float32), 5)
    assert m.sum() == 5


def test_k_rounding():
    # k = floor(rho n + 1/2): round half up of rho n
    assert oracle.k_of(0.5, 7) == 4
    assert oracle.k_of(0.05, 3) == 0
    assert oracle.k_of(0.1, 1024 * 1024) == 104858
    assert oracle.k_of(0.05, 1536 * 1536) == 117965
    assert oracle.k_of(1.0, 5) == 5 and oracle.k_of(0.0, 5) == 0
    assert oracle.k_of(1.5, 5) == 5


def test_block_units_order_and_edges():
    u = oracle.block_units(5, 7, 2, 3)
    assert len(u) == 3 * 3
    assert u[0].tolist() == [0, 1, 2, 7, 8, 9]
    assert u[2].tolist() == [6, 13]            # partial edge block
    assert u[8].tolist() == [34]
    allidx = np.sort(np.concatenate(u))
    assert np.array_equal(allidx, np.arange(35))


def test_global_scope_is_concatenation():
    rng = np.random.default_rng(3)
    a = rng.normal(0, 1, (3, 4)).astype(np.float32)
    b = rng.normal(0, 1, 5).astype(np.float32)
    masks, st = oracle.topk_masks([a, b], [(3, 4), (1, 5)], 0.3, oracle.SCOPE_GLOBAL)
    cat = np.concatenate([a.ravel(), b])
    ref = _sort_reference(cat, oracle.k_of(0.3, 17))
    assert np.array_equal(np.concatenate(masks), ref)
    assert st.shape == (1,)


# ---------------------------------------------------------------------------
# encodings
# ---------------------------------------------------------------------------

def test_f32_to_bf16_matches_library():
    rng = np.random.default_rng(11)
    bits = rng.integers(0, 2**32, 2_000_000, dtype=np.uint64).astype(np.uint32)
    edge = np.array([0, 0x80000000, 0x3F808000, 0x3F818000, 0x3F80FFFF, 0x7F7FFFFF,
                     0x7F7F8000, 0x00008000, 0x00018000, 0x007FFFFF, 0x7F800000, 0xFF800000],
                    np.uint32)
    bits = np.concatenate([bits, edge])
    x = bits.view(np.float32)
    finite = np.isfinite(x)
    ref = torch.from_numpy(x[finite].copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.f32_to_bf16(x[finite])
    np.testing.assert_array_equal(got, ref)


def _bf16_value(b):
    return Fraction(float(np.uint32(int(b) << 16).view(np.float32)))


def test_f64_to_bf16_one_rounding():
    rng = np.random.default_rng(5)
    xs = list(rng.normal(0, 0.02, 3000)) + list(rng.normal(0, 1e-30, 200)) + \
         [1 + 2**-8, 1 + 3 * 2**-8, 1 + 2**-8 + 2**-40, -(1 + 2**-8), 2**-133, 2**-134,
          3 * 2**-135, 1e-45, 3.3e38, 3.4e38]
    got = oracle.f64_to_bf16(np.array(xs))
    for x, b in zip(xs, got):
        # exact nearest-even among all finite bfloat16 values, by rational arithmetic
        fx = Fraction(x)
        f32b = int(np.float32(abs(x)).view(np.uint32)) >> 16
        cands = [c for c in range(max(0, f32b - 2), min(0x7F7F, f32b + 2) + 1)]
        best = min(cands, key=lambda c: (abs(_bf16_value(c) - abs(fx)), c & 1))
        # IEEE overflow: at or beyond max + half an ulp = (2 - 2^-8) 2^127 -> infinity
        if abs(fx) >= Fraction(2**127) * (2 - Fraction(1, 256)):
            best = 0x7F80
        want = best | (0x8000 if x < 0 else 0)
        assert int(b) == want, (x, hex(int(b)), hex(want))


def test_bf16_roundtrip_exact():
    b = np.arange(0, 0x7F80, dtype=np.uint16)
    f = oracle.bf16_to_f32(b)
    np.testing.assert_array_equal(oracle.f32_to_bf16(f), b)
    np.testing.assert_array_equal(oracle.f64_to_bf16(f.astype(np.float64)), b)


# ---------------------------------------------------------------------------
# merge operators: closed forms and invariants
# ---------------------------------------------------------------------------

def _rand_set(rng, shapes, scale=1e-3, dtype="bf16"):
    th0, tau = [], []
    for s in shapes:
        w = rng.normal(0, 0.02, s).astype(np.float32)
        t = rng.normal(0, scale, s).astype(np.float32)
        th0.append(oracle.f32_to_bf16(w) if dtype == "bf16" else w)
        tau.append(t)
    return th0, tau


def test_rho_one_reduces_ties_and_iso():
    rng = np.random.default_rng(1)
    th0, tau = _rand_set(rng, [(16, 24)], dtype="f32")
    r_t = oracle.merge(th0, [tau], oracle.TIES, density=1.0, lam=0.7, is_1d=[False])
    r_a = oracle.merge(th0, [tau], oracle.TA, lam=0.7, is_1d=[False])
    np.testing.assert_array_equal(r_t["out64"][0], r_a["out64"][0])
    np.testing.assert_array_equal(r_t["out64"][0],
                                  th0[0].astype(np.float64).ravel() + 0.7 * tau[0].astype(np.float64).ravel())
    r_i = oracle.merge(th0, [tau], oracle.ISO, density=1.0, is_1d=[False])
    G = float(np.sum(tau[0].astype(np.float64) ** 2))
    assert r_i["gram"][0][0, 0] == pytest.approx(G, rel=1e-15)
    assert r_i["coef"][0][0] == pytest.approx(G / (G + 1e-12), rel=1e-15)


@pytest.mark.parametrize("op", [oracle.TA, oracle.TIES, oracle.ISO])
def test_zero_delta_fixed_point(op):
    rng = np.random.default_rng(2)
    th0, _ = _rand_set(rng, [(8, 32), (1, 32)])
    th0[0].ravel()[5] = 0x8000  # -0.0 base weight keeps its sign
    zeros = [np.zeros(a.shape, np.float32) for a in th0]
    r = oracle.merge(th0, [zeros, zeros, zeros], op, density=0.2, is_1d=[False, True])
    for a, b in zip(r["out"], th0):
        np.testing.assert_array_equal(a, b)


def test_identical_experts():
    rng = np.random.default_rng(4)
    th0, tau = _rand_set(rng, [(32, 32)], dtype="f32")
    K = 3
    r = oracle.merge(th0, [tau] * K, oracle.TIES, density=0.2, lam=1.0, is_1d=[False])
    m, _ = oracle.topk_unit(tau[0].ravel(), oracle.k_of(0.2, 1024))
    want = th0[0].ravel().astype(np.float64) + m * tau[0].ravel().astype(np.float64)
    np.testing.assert_allclose(r["out64"][0], want, rtol=0, atol=1e-15)
    r = oracle.merge(th0, [tau] * K, oracle.ISO, density=0.2, is_1d=[False])
    G = r["gram"][0][0, 0]
    # (G 1 1^T + ridge I) c = G 1  ->  c_i = G / (K G + ridge).  The system has
    # condition number ~ K G / ridge, so each c_i is fixed only to ~cond * eps,
    # while sum(c) (along the well-conditioned eigenvector 1) is fixed to eps.
    assert np.sum(r["coef"][0]) == pytest.approx(K * G / (K * G + 1e-12), rel=1e-12)
    np.testing.assert_allclose(r["coef"][0], G / (K * G + 1e-12), rtol=1e-6)
    # sum(c) = 1 - ridge / (K G) + ...: the update is the trimmed delta up to ~1e-8 of it
    np.testing.assert_allclose(r["out64"][0], want, rtol=0, atol=1e-8 * np.abs(tau[0]).max())


def test_disjoint_supports():
    rng = np.random.default_rng(6)
    n = 400
    t1 = np.zeros(n, np.float32)
    t2 = np.zeros(n, np.float32)
    t1[:200] = rng.normal(0, 1e-3, 200)
    t2[200:] = rng.normal(0, 1e-3, 200)
    th0 = rng.normal(0, 0.02, n).astype(np.float32).reshape(1, n)
    r = oracle.merge([th0], [[t1.reshape(1, n)], [t2.reshape(1, n)]], oracle.ISO,
                     density=0.5, is_1d=[False])
    G = r["gram"][0]
    assert G[0, 1] == 0.0 and G[1, 0] == 0.0
    np.testing.assert_allclose(r["coef"][0], np.diag(G) / (np.diag(G) + 1e-12), rtol=1e-15)
    rt = oracle.merge([th0], [[t1.reshape(1, n)], [t2.reshape(1, n)]], oracle.TIES,
                      density=0.5, is_1d=[False])
    # disjoint supports never conflict: TIES keeps each trimmed entry as is, and
    # ISO's c_i = G_ii / (G_ii + ridge) differs from 1 by ~ridge / G_ii ~ 1e-8
    np.testing.assert_allclose(r["out64"][0], rt["out64"][0], rtol=0,
                               atol=1e-7 * max(np.abs(t1).max(), np.abs(t2).max()))


def test_anticorrelated_clips_and_cancels():
    rng = np.random.default_rng(8)
    th0, tau = _rand_set(rng, [(16, 16)])
    neg = [-t for t in tau]
    r = oracle.merge(th0, [tau, neg], oracle.ISO, density=0.3, is_1d=[False])
    np.testing.assert_array_equal(r["coef"][0], [1.5, 1.5])   # ridge-dominated, clipped
    np.testing.assert_array_equal(r["out"][0], th0[0])
    rt = oracle.merge(th0, [tau, neg], oracle.TIES, density=0.3, is_1d=[False])
    np.testing.assert_array_equal(rt["out"][0], th0[0])       # every election cancels


def test_retention_matches_library_solve():
    rng = np.random.default_rng(9)
    for K in range(1, 9):
        A = rng.normal(0, 1, (K, 40))
        A[rng.random(K) < 0.2] = 0.0                 # zero-norm experts are dropped
        G = A @ A.T
        c = oracle.retention(G, ridge=1e-12, c_min=0.0, c_max=1.5)
        keep = np.diag(G) > 0
        want = np.zeros(K)
        if keep.any():
            Gi = G[np.ix_(keep, keep)]
            want[keep] = np.clip(np.linalg.solve(Gi + 1e-12 * np.eye(Gi.shape[0]), np.diag(Gi)), 0, 1.5)
        np.testing.assert_allclose(c, want, rtol=1e-9, atol=1e-12)


def test_ties_election_and_disjoint_mean_small():
    # one coordinate, three experts, every mask on: +3, -1, +1 -> gamma + -> mean(3, 1) = 2
    th0 = np.zeros((1, 1), np.float32)
    ex = [[np.full((1, 1), v, np.float32)] for v in (3.0, -1.0, 1.0)]
    r = oracle.merge([th0], ex, oracle.TIES, density=1.0, lam=0.5, is_1d=[False])
    assert r["out64"][0][0] == 1.0                    # 0.5 * mean(3, 1)
    ex = [[np.full((1, 1), v, np.float32)] for v in (-3.0, 1.0, 1.0)]
    r = oracle.merge([th0], ex, oracle.TIES, density=1.0, lam=1.0, is_1d=[False])
    assert r["out64"][0][0] == -3.0                   # sum -1 -> gamma -, A = {1}


def test_permuting_experts_keeps_masks_and_merge():
    rng = np.random.default_rng(10)
    th0, t1 = _rand_set(rng, [(20, 20)])
    _, t2 = _rand_set(rng, [(20, 20)])
    _, t3 = _rand_set(rng, [(20, 20)])
    for op in (oracle.TA, oracle.TIES, oracle.ISO):
        a = oracle.merge(th0, [t1, t2, t3], op, density=0.2, is_1d=[False])
        b = oracle.merge(th0, [t3, t1, t2], op, density=0.2, is_1d=[False])
        np.testing.assert_allclose(a["out64"][0], b["out64"][0], rtol=1e-12, atol=1e-15)
        if op != oracle.TA:
            assert np.array_equal(a["masks"][0][0], b["masks"][1][0])


def test_checkpoint_delta_exact_for_bf16():
    rng = np.random.default_rng(12)
    th0 = oracle.f32_to_bf16(rng.normal(0, 0.02, 5000).astype(np.float32))
    th1 = oracle.f32_to_bf16(oracle.bf16_to_f32(th0) + rng.normal(0, 5e-4, 5000).astype(np.float32))
    t32, t64 = oracle.delta(th1, th0)
    np.testing.assert_array_equal(t32.astype(np.float64), t64)
    # K = 1, rho = 1, lambda = 1: the update reproduces the checkpoint bit for bit
    r = oracle.update([th0.reshape(50, 100)], [th1.reshape(50, 100)], oracle.TIES,
                      density=1.0, lam=1.0, is_1d=[False])
    np.testing.assert_array_equal(r["out"][0].ravel(), th1)


def test_ties_election_uses_trimmed_vectors():
    # App. F elects gamma^p = sign(sum_i trimmed tau_i^p).  Two coordinates,
    # density 1/2 (k = 1 each): tau1 = [1, 5] keeps p1; tau2 = [-1/2, 1/10] keeps p0.
    # At p0 the trimmed sum is -1/2 (gamma -, merged -1/2); the untrimmed sum
    # would be +1/2 and would leave an empty agreeing set.
    th0 = np.zeros((1, 2), np.float32)
    t1 = np.array([[1.0, 5.0]], np.float32)
    t2 = np.array([[-0.5, 0.1]], np.float32)
    r = oracle.merge([th0], [[t1], [t2]], oracle.TIES, density=0.5, lam=1.0, is_1d=[False])
    assert r["out64"][0][0] == -0.5
    assert r["out64"][0][1] == 5.0


def test_ties_untrimmed_tensor_keeps_every_entry():
    # mask_1d = 0: a 1-D tensor enters TIES untrimmed (m_i = 1 everywhere); with
    # K = 1 the merge is then theta_0 + lambda tau on every entry.
    rng = np.random.default_rng(13)
    th0 = rng.normal(0, 0.02, 64).astype(np.float32)
    tau = rng.normal(0, 1e-3, 64).astype(np.float32)
    r = oracle.merge([th0], [[tau]], oracle.TIES, density=0.1, lam=1.0, mask_1d=False, is_1d=[True])
    np.testing.assert_array_equal(r["out64"][0], th0.astype(np.float64) + tau.astype(np.float64))
    r = oracle.merge([th0], [[tau]], oracle.TIES, density=0.1, lam=1.0, mask_1d=True, is_1d=[True])
    assert (r["out64"][0] != th0.astype(np.float64)).sum() == oracle.k_of(0.1, 64)


# ---------------------------------------------------------------------------
# RAM (App. F): activity threshold, unique values kept, shared ones averaged
# over the active experts only
# ---------------------------------------------------------------------------

class TestRamHandWorked:
    g = _golden("handworked_ram_k3_1x8.json")

    def _run(self, op, **kw):
        th0 = _f32(self.g["theta0"]).reshape(1, 8)
        taus = [[_f32(_fr(self.g[f"tau{i}"])).reshape(1, 8)] for i in (1, 2, 3)]
        return oracle.merge([th0], taus, op, lam=1.0, is_1d=[False],
                            eps_act=float(Fraction(self.g["eps_act"])), **kw)

    def test_ram(self):
        r = self._run(oracle.RAM)
        want = [Fraction(x) for x in self.g["ram"]]
        got = r["out64"][0]
        for p, w in enumerate(want):
            # binary64 mean of at most three dyadic values: exact except the
            # one division by c, which rounds once
            assert got[p] == pytest.approx(float(w), rel=2 ** -52, abs=0), p
        # the entries with a dyadic result are exact
        for p in (0, 1, 2, 4, 5):
            assert got[p] == float(want[p])
        assert r["units"].size == 0   # RAM trims nothing

    def test_ta_differs_where_ram_keeps_or_drops(self):
        r = self._run(oracle.TA)
        np.testing.assert_array_equal(r["out64"][0], _fr(self.g["ta"]))


def _ram_exact(th0, taus, eps, lam):
    """RAM evaluated in exact rationals, entry by entry (App. F coordinate rule)."""
    out = []
    for p in range(th0.size):
        act = [Fraction(float(t[p])) for t in taus if abs(float(t[p])) > eps]
        c = len(act)
        m = Fraction(0) if c == 0 else (act[0] if c == 1 else sum(act, Fraction(0)) / c)
        out.append(Fraction(float(th0[p])) + Fraction(lam) * m)
    return out


@pytest.mark.parametrize("K,lam", [(2, 1.0), (3, 0.5), (5, 1.0), (8, 0.75)])
def test_ram_brute_force_rationals(K, lam):
    rng = np.random.default_rng(100 + K)
    n = 300
    eps = float(np.float32(1e-3))
    th0 = rng.normal(0, 0.02, n).astype(np.float32)
    taus = []
    for i in range(K):
        t = rng.normal(0, 1e-3, n).astype(np.float32)
        t[rng.random(n) < 0.3] = 0.0
        t[rng.random(n) < 0.05] = np.float32(eps) * rng.choice([-1, 1], n)[0]   # on the threshold
        taus.append(t)
    r = oracle.merge([th0.reshape(1, n)], [[t.reshape(1, n)] for t in taus], oracle.RAM,
                     lam=lam, is_1d=[False], eps_act=eps)
    want = _ram_exact(th0, taus, eps, lam)
    got = r["out64"][0]
    for p in range(n):
        assert got[p] == pytest.approx(float(want[p]), rel=4e-16, abs=1e-300), p


def test_ram_disjoint_supports_is_task_arithmetic():
    rng = np.random.default_rng(110)
    n, K = 512, 4
    th0 = rng.normal(0, 0.02, n).astype(np.float32).reshape(1, n)
    owner = rng.integers(0, K, n)
    taus = []
    for i in range(K):
        t = np.zeros(n, np.float32)
        sel = owner == i
        # every owned entry well above the threshold, either sign
        t[sel] = np.sign(rng.normal(size=sel.sum())) * (np.abs(rng.normal(0, 1e-3, sel.sum())) + 1e-4)
        taus.append(t.reshape(1, n))
    r = oracle.merge([th0], [[t] for t in taus], oracle.RAM, lam=1.0, is_1d=[False],
                     eps_act=float(np.float32(1e-5)))
    ra = oracle.merge([th0], [[t] for t in taus], oracle.TA, lam=1.0, is_1d=[False])
    # one active expert per entry: its value is kept whole, as TA's sum gives it
    np.testing.assert_array_equal(r["out64"][0], ra["out64"][0])


@pytest.mark.parametrize("K", [2, 4, 8])
def test_ram_identical_experts_keep_the_task_vector(K):
    rng = np.random.default_rng(120 + K)
    th0, tau = _rand_set(rng, [(16, 40)], dtype="f32")
    r = oracle.merge(th0, [tau] * K, oracle.RAM, lam=1.0, is_1d=[False], eps_act=0.0)
    t = tau[0].ravel().astype(np.float64)
    want = np.where(t == 0.0, th0[0].ravel().astype(np.float64), th0[0].ravel().astype(np.float64) + t)
    # K copies of one value sum exactly for K a power of two; the mean is the value
    np.testing.assert_array_equal(r["out64"][0], want)


def test_ram_threshold_above_every_update_is_fixed_point():
    rng = np.random.default_rng(130)
    th0, tau = _rand_set(rng, [(8, 32), (1, 32)])
    th0[0].ravel()[3] = 0x8000   # -0.0 keeps its sign
    eps = max(float(np.abs(oracle.load(t)[0]).max()) for t in tau)
    r = oracle.merge(th0, [tau, tau], oracle.RAM, is_1d=[False, True], eps_act=eps)
    for a, b in zip(r["out"], th0):
        np.testing.assert_array_equal(a, b)


def test_ram_single_expert_is_a_threshold_mask():
    rng = np.random.default_rng(140)
    n = 2000
    th0 = rng.normal(0, 0.02, n).astype(np.float32).reshape(1, n)
    t = rng.normal(0, 1e-5, n).astype(np.float32).reshape(1, n)
    eps = float(np.float32(1e-5))
    r = oracle.update([th0], [t], oracle.RAM, update_is_delta=True, is_1d=[False], eps_act=eps)
    tt = t.ravel().astype(np.float64)
    want = np.where(np.abs(tt) > eps, th0.ravel().astype(np.float64) + tt, th0.ravel().astype(np.float64))
    np.testing.assert_array_equal(r["out64"][0], want)
    assert 0 < np.sum(np.abs(tt) > eps) < n


def test_f32_to_bf16_exhaustive():
    """Every binary32 bit pattern but the NaNs: the oracle's bit-level
    round-to-nearest-even against torch's conversion, 2^24 patterns at a
    time in reused buffers."""
    import ctypes
    lib = oracle._lib()
    CH = 1 << 24
    idx = np.arange(CH, dtype=np.uint32)
    bits = np.empty(CH, np.uint32)
    got = np.empty(CH, np.uint16)
    want = torch.empty(CH, dtype=torch.bfloat16)
    P = ctypes.c_void_p
    for c in range(1 << 8):
        np.add(idx, np.uint32(c * CH), out=bits)
        x = bits.view(np.float32)
        lib.orc_f32_to_bf16_array(P(x.ctypes.data), CH, P(got.ctypes.data))
        want.copy_(torch.from_numpy(x))
        w = want.view(torch.int16).numpy().view(np.uint16)
        ok = (got == w) | np.isnan(x)
        if not ok.all():
            i = int(np.flatnonzero(~ok)[0])
            raise AssertionError(f"pattern {bits[i]:#010x}: oracle {got[i]:#06x}, torch {w[i]:#06x}")
