"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Masks, thresholds and tie counts must match bit for bit; merged and updated
values within the tolerances stated in parity_util.  Inputs are seeded and
synthetic (synth), shaped like the paper's workloads but small enough for the
oracle, with several tiles per tensor and ragged tails.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_19331_gb300 as iso
import synth
from paper_2607_19331_gb300 import _abi
from parity_util import assert_units_equal, assert_values_close, to_np, unpack_mask

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()


OPS = {"ta": oracle.TA, "ties": oracle.TIES, "iso": oracle.ISO}
OP_NAME = {oracle.TA: "ta", oracle.TIES: "ties", oracle.ISO: "iso", oracle.RAM: "ram"}
SCOPES = {"tensor": oracle.SCOPE_TENSOR, "block": oracle.SCOPE_BLOCK, "global": oracle.SCOPE_GLOBAL}

# several tiles and ragged tails, partial 128 x 128 blocks, 1-D, tiny and empty
MIXED = [(300, 1000, False), (257, 129, False), (1, 1536, True), (3, 7, False),
         (0, 5, False), (64, 4096, False), (1, 5, True), (40, 1000, False)]


def _np_list(ts):
    return [to_np(t) for t in ts]


def _shapes(shapes):
    return [(r, c) for r, c, _ in shapes]


def _is1d(shapes):
    return [o for _, _, o in shapes]


def _taus(shapes, seed, dtype, ties=False):
    out = []
    for q, s in enumerate(shapes):
        g = torch.Generator().manual_seed(seed * 131 + q)
        r, c, one = s
        x = torch.randn(r * c, generator=g) * 1e-3
        if ties:   # coarse grid: thousands of exact ties
            x = torch.round(x * 4000) / 4000
        x = x.reshape(c) if one else x.reshape(r, c)
        out.append(x.to(dtype))
    return out


# ---------------------------------------------------------------------------
# TopKMask
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("scope", ["tensor", "block", "global"])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("density", [0.0, 0.01, 0.05, 0.2, 0.5, 1.0])
def test_topk_mask_parity(scope, dtype, density):
    taus = _taus(MIXED, 1, dtype, ties=(dtype == torch.float32 and density == 0.2))
    dev = [t.to(DEV) for t in taus]
    masks, st = iso.iso_topk_mask(dev, density=density, scope=scope, stats=True)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    t32 = [oracle.load(to_np(t))[0] for t in taus]
    om, ou = oracle.topk_masks(t32, _shapes(MIXED), density, SCOPES[scope])
    for q, (m, t) in enumerate(zip(masks, taus)):
        got = unpack_mask(m, t.numel())
        assert np.array_equal(got, om[q]), f"mask of tensor {q} differs ({scope}, {density})"
    assert_units_equal(st.units_numpy()[0], ou, f"units {scope} {density}")


def test_topk_mask_bf16_checkpoint_ties():
    # bfloat16-quantised RL deltas: the threshold sits inside a run of exact ties
    shapes = [(512, 768, False), (96, 2048, False)]
    th0, th1 = synth.rl_update_set(shapes, seed=3)
    taus = [(a.float() - b.float()) for a, b in zip(th1, th0)]
    dev = [t.to(DEV) for t in taus]
    for density in (0.05, 0.2):
        masks, st = iso.iso_topk_mask(dev, density=density, scope="tensor", stats=True)
        om, ou = oracle.topk_masks([to_np(t) for t in taus], _shapes(shapes), density)
        for q, (m, t) in enumerate(zip(masks, taus)):
            assert np.array_equal(unpack_mask(m, t.numel()), om[q])
        u = st.units_numpy()[0]
        assert_units_equal(u, ou)
        assert (u["ties_at_thresh"] > u["ties_taken"]).all()   # partial ties really exercised


def test_band_miss_falls_back_exactly():
    # Zero every entry the band sample reads and make the rest large: the band
    # misses and the unit is resolved by the full-data radix select.
    n = 300_000
    x = (torch.arange(n, dtype=torch.float32) % 977 + 1.0) * 1e-3
    S, C = 24576, 256   # the library's sample size and chunk length
    nch = S // C
    for c in range(nch):
        p = int((n - C) * c / (nch - 1))
        x[p:p + C] = 0.0
    t = x.reshape(300, 1000)
    masks, st = iso.iso_topk_mask([t.to(DEV)], density=0.1, scope="tensor", stats=True)
    u = st.units_numpy()[0]
    assert u["flags"][0] & 1, "expected the fallback path"
    om, ou = oracle.topk_masks([t.numpy()], [(300, 1000)], 0.1)
    assert np.array_equal(unpack_mask(masks[0], n), om[0])
    assert_units_equal(u, ou)


# ---------------------------------------------------------------------------
# updates and merges
# ---------------------------------------------------------------------------
def _check_merge(res_gpu, st, r_orc, theta0, op, K, check_units=True, what=""):
    for q, (o, b) in enumerate(zip(res_gpu, theta0)):
        g = to_np(o)
        assert g.dtype == (np.uint16 if b.dtype == torch.bfloat16 else np.float32)
        assert_values_close(g, r_orc["out64"][q], r_orc["mag"][q], f"{what} tensor {q}",
                            op=OP_NAME[op], K=K)
    if st is None:
        return
    assert int(st.status.item()) == 0
    if check_units and op != oracle.TA:
        assert_units_equal(st.units_numpy(), r_orc["units"], what)
    if op == oracle.ISO:
        coef = st.coef.cpu().numpy()[: len(theta0) * K].reshape(len(theta0), K)
        gram = st.gram.cpu().numpy()[: len(theta0) * K * K].reshape(len(theta0), K, K)
        for q in range(len(theta0)):
            np.testing.assert_allclose(gram[q], r_orc["gram"][q], rtol=2e-6,
                                       atol=2e-6 * np.abs(r_orc["gram"][q]).max() + 1e-300)
            np.testing.assert_allclose(coef[q], r_orc["coef"][q], rtol=1e-5, atol=1e-9)


MINI = synth.qwen_shapes("qwen1.5b", layers=2, scale=8)


@pytest.mark.parametrize("scope", ["tensor", "block", "global"])
@pytest.mark.parametrize("op", ["iso", "ties", "ta"])
def test_update_checkpoint_bf16(scope, op):
    th0, th1 = synth.rl_update_set(MINI, seed=0)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    out, st = iso.iso_update(d0, d1, op=op, update_is_delta=False, density=0.05, scope=scope,
                             lam=1.0, stats=True)
    torch.cuda.synchronize()
    r = oracle.update(_np_list(th0), _np_list(th1), OPS[op], update_is_delta=False, density=0.05,
                      scope=SCOPES[scope], lam=1.0, shapes=_shapes(MINI), is_1d=_is1d(MINI))
    _check_merge(out, st, r, th0, OPS[op], 1, what=f"update {op} {scope}")


@pytest.mark.parametrize("op", ["iso", "ties"])
def test_block_update_many_full_units(op):
    # more 128 x 128 units than SMs: each persistent block-select CTA walks
    # several consecutive units, prefetching the next full unit, across tensor
    # boundaries, partial edge units and a 1-D tensor
    shapes = [(1024, 2048, False), (300, 1000, False), (2048, 1024, False), (1, 2048, True),
              (640, 768, False)]
    th0, th1 = synth.rl_update_set(shapes, seed=3)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    out, st = iso.iso_update(d0, d1, op=op, update_is_delta=False, density=0.05, scope="block",
                             lam=1.0, stats=True)
    torch.cuda.synchronize()
    r = oracle.update(_np_list(th0), _np_list(th1), OPS[op], update_is_delta=False, density=0.05,
                      scope=oracle.SCOPE_BLOCK, lam=1.0, shapes=_shapes(shapes), is_1d=_is1d(shapes))
    _check_merge(out, st, r, th0, OPS[op], 1, what=f"block update {op}")


@pytest.mark.parametrize("op", ["ta", "ties", "iso"])
def test_tiny_fp32_k2(op):
    # 1024 x 1024 fp32 base, K = 2 fp32 task vectors, density 10 %, lambda 1, seed 0
    th0, taus = synth.tiny_set(seed=0)
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in taus]
    out, st = iso.iso_merge(d0, dx, op=op, experts_are_deltas=True, density=0.1, lam=1.0, stats=True)
    torch.cuda.synchronize()
    r = oracle.merge(_np_list(th0), [_np_list(e) for e in taus], OPS[op], density=0.1, lam=1.0,
                     is_1d=[False])
    _check_merge(out, st, r, th0, OPS[op], 2, what=f"tiny {op}")


@pytest.mark.parametrize("scope", ["tensor", "block", "global"])
@pytest.mark.parametrize("op", ["ties", "iso", "ta"])
@pytest.mark.parametrize("K", [3, 8])
def test_merge_bf16_base_fp32_deltas(scope, op, K):
    shapes = synth.qwen_shapes("qwen1.5b", layers=1, scale=8)
    th0 = synth.base_weights(shapes, seed=5)
    taus, _ = synth.merge_experts(shapes, seed=5, K=K)
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in taus]
    out, st = iso.iso_merge(d0, dx, op=op, density=0.1, scope=scope, lam=0.7, stats=True)
    torch.cuda.synchronize()
    r = oracle.merge(_np_list(th0), [_np_list(e) for e in taus], OPS[op], density=0.1,
                     scope=SCOPES[scope], lam=0.7, shapes=_shapes(shapes), is_1d=_is1d(shapes))
    _check_merge(out, st, r, th0, OPS[op], K, what=f"merge K={K} {op} {scope}")


@pytest.mark.parametrize("scope", ["tensor", "block", "global"])
@pytest.mark.parametrize("op", ["ties", "iso", "ta"])
@pytest.mark.parametrize("K,experts", [(2, "delta_bf16"), (4, "ckpt_bf16"), (5, "delta_bf16"),
                                       (5, "ckpt_f32"), (7, "delta_f32")])
def test_merge_expert_counts_and_dtypes(scope, op, K, experts):
    # every compile-time expert bound (2, 4, 8) with K below and at it, bf16
    # and fp32 experts given as task vectors or as checkpoints, on shapes with
    # ragged tails, 1-D tensors, partial blocks and an empty tensor
    shapes = MIXED
    base_dt = torch.float32 if experts == "ckpt_f32" else torch.bfloat16
    th0 = synth.base_weights(shapes, seed=11, dtype=base_dt)
    xs = []
    for i in range(K):
        d = _taus(shapes, 40 + i, torch.float32, ties=(i % 2 == 1))
        if experts == "delta_bf16":
            xs.append([x.to(torch.bfloat16) for x in d])
        elif experts == "delta_f32":
            xs.append(d)
        else:
            dt = torch.bfloat16 if experts == "ckpt_bf16" else torch.float32
            xs.append([(b.float() + x).to(dt) for b, x in zip(th0, d)])
    is_delta = experts.startswith("delta")
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in xs]
    out, st = iso.iso_merge(d0, dx, op=op, experts_are_deltas=is_delta, density=0.15, scope=scope,
                            lam=0.9, stats=True)
    torch.cuda.synchronize()
    r = oracle.merge(_np_list(th0), [_np_list(e) for e in xs], OPS[op], experts_are_deltas=is_delta,
                     density=0.15, scope=SCOPES[scope], lam=0.9, shapes=_shapes(shapes),
                     is_1d=_is1d(shapes))
    _check_merge(out, st, r, th0, OPS[op], K, what=f"merge K={K} {experts} {op} {scope}")


def test_merge_checkpoints_mask_1d_off():
    shapes = MIXED
    th0 = synth.base_weights(shapes, seed=9, dtype=torch.float32)
    ck = []
    for i in range(2):
        d = _taus(shapes, 20 + i, torch.float32)
        ck.append([(a + b) for a, b in zip(th0, d)])
    d0 = [t.to(DEV) for t in th0]
    dx = [[t.to(DEV) for t in e] for e in ck]
    out, st = iso.iso_merge(d0, dx, op="ties", experts_are_deltas=False, density=0.3,
                            mask_1d=False, stats=True)
    torch.cuda.synchronize()
    r = oracle.merge(_np_list(th0), [_np_list(e) for e in ck], oracle.TIES, experts_are_deltas=False,
                     density=0.3, mask_1d=False, shapes=_shapes(shapes), is_1d=_is1d(shapes))
    _check_merge(out, st, r, th0, oracle.TIES, 2, what="ties checkpoints mask_1d=0")


@pytest.mark.parametrize("scope", ["tensor", "block", "global"])
def test_update_mask_1d_off(scope):
    # TIES leaving 1-D tensors untrimmed in a K = 1 update: outside the
    # selection every entry is kept (GLOBAL scope: outside the one unit, whose
    # positions count only the trimmed tensors)
    th0, th1 = synth.rl_update_set(MINI, seed=12)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    out, st = iso.iso_update(d0, d1, op="ties", update_is_delta=False, density=0.05, scope=scope,
                             lam=1.0, mask_1d=False, stats=True)
    torch.cuda.synchronize()
    r = oracle.update(_np_list(th0), _np_list(th1), oracle.TIES, update_is_delta=False, density=0.05,
                      scope=SCOPES[scope], lam=1.0, mask_1d=False, shapes=_shapes(MINI), is_1d=_is1d(MINI))
    _check_merge(out, st, r, th0, oracle.TIES, 1, what=f"update ties mask_1d=0 {scope}")


# ---------------------------------------------------------------------------
# edge cases
# ---------------------------------------------------------------------------
def test_zero_delta_is_fixed_point():
    th0 = synth.base_weights(MIXED, seed=2)
    th0[0].view(-1)[7] = -0.0
    zeros = [torch.zeros(t.shape, dtype=torch.float32) for t in th0]
    d0 = [t.to(DEV) for t in th0]
    for op in ("ta", "ties", "iso"):
        out = iso.iso_merge(d0, [[z.to(DEV) for z in zeros]] * 2, op=op, density=0.2)
        for a, b in zip(out, d0):
            assert torch.equal(a.view(torch.int16), b.view(torch.int16)), op


def test_in_place_update_and_determinism():
    th0, th1 = synth.rl_update_set(MINI, seed=4)
    d1 = [t.to(DEV) for t in th1]
    a = iso.iso_update([t.to(DEV) for t in th0], d1, op="iso", density=0.05)
    b = iso.iso_update([t.to(DEV) for t in th0], d1, op="iso", density=0.05)
    inplace = [t.to(DEV) for t in th0]
    iso.iso_update(inplace, d1, op="iso", density=0.05, out=inplace)
    for x, y, z in zip(a, b, inplace):
        assert torch.equal(x.view(torch.int16), y.view(torch.int16))
        assert torch.equal(x.view(torch.int16), z.view(torch.int16))


def test_small_workspace_groups_give_same_result():
    th0, th1 = synth.rl_update_set(MINI, seed=6)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    cfg = iso.merge_cfg("iso", 0.05)
    mn, full = iso.iso_workspace_size(d0, 1, cfg)
    assert mn < full
    ref, st_ref = iso.iso_update(d0, d1, op="iso", density=0.05, stats=True)
    got, st = iso.iso_update(d0, d1, op="iso", density=0.05, stats=True, ws_bytes=mn,
                             workspace=iso.Workspace(DEV))
    for x, y in zip(ref, got):
        assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    u, u_ref = st.units_numpy(), st_ref.units_numpy()
    assert_units_equal(u, u_ref, "grouped vs whole")
    assert np.array_equal(u["flags"], u_ref["flags"]), "a unit took the fallback in one run only"
    with pytest.raises(iso.IsoError) as e:
        iso.iso_update(d0, d1, op="iso", density=0.05, ws_bytes=mn - 256, workspace=iso.Workspace(DEV))
    assert e.value.code == _abi.ISO_ERR_WORKSPACE


def test_nonfinite_input_reported():
    th0, th1 = synth.rl_update_set(MINI[:3], seed=7)
    th1[1].view(-1)[123] = float("nan")
    _, st = iso.iso_update([t.to(DEV) for t in th0], [t.to(DEV) for t in th1], op="ties",
                           density=0.05, stats=True)
    torch.cuda.synchronize()
    assert int(st.status.item()) == _abi.ISO_ERR_NONFINITE


def test_argument_errors():
    a = torch.zeros(64, 64, dtype=torch.bfloat16, device=DEV)
    b = torch.zeros(64, 32, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(iso.IsoError) as e:
        iso.iso_update([a], [b], op="ties")
    assert e.value.code == _abi.ISO_ERR_SHAPE
    big = torch.zeros(64 * 64 + 8, dtype=torch.bfloat16, device=DEV)
    mis = big[1:1 + 64 * 64].view(64, 64)
    with pytest.raises(iso.IsoError) as e:
        iso.iso_update([a], [mis], op="ties")
    assert e.value.code == _abi.ISO_ERR_ALIGN
    with pytest.raises(iso.IsoError) as e:
        iso.iso_update([a], [a.clone()], op="ties", density=1.5)
    assert e.value.code == _abi.ISO_ERR_ARG
    c = torch.zeros(64, 64, dtype=torch.float32, device=DEV)
    with pytest.raises(iso.IsoError) as e:
        iso.iso_merge([a], [[a.clone()]], out=[c])
    assert e.value.code == _abi.ISO_ERR_DTYPE


def test_delta_parity():
    th0, th1 = synth.rl_update_set(MIXED, seed=8)
    tau = iso.iso_delta([t.to(DEV) for t in th1], [t.to(DEV) for t in th0])
    torch.cuda.synchronize()
    for t, a, b in zip(tau, th1, th0):
        t32, _ = oracle.delta(to_np(a), to_np(b))
        assert np.array_equal(to_np(t).view(np.uint32), t32.view(np.uint32))


def test_launch_counter_moves():
    n0 = iso.launch_count()
    th0, th1 = synth.rl_update_set(MINI[:4], seed=1)
    iso.iso_update([t.to(DEV) for t in th0], [t.to(DEV) for t in th1], op="iso", density=0.05)
    assert iso.launch_count() > n0


# ---------------------------------------------------------------------------
# full size, sampled: the Qwen2.5-1.5B-shaped update in the benchmark's launch
# configuration, checked tensor by tensor on a sample of every shape class
# ---------------------------------------------------------------------------
def test_full_size_qwen15b_update_sampled():
    shapes = synth.qwen_shapes("qwen1.5b")
    th0, th1 = synth.rl_update_set(shapes, seed=0, device=DEV)
    ws = iso.Workspace(DEV)
    out, st = iso.iso_update(th0, th1, op="iso", density=0.05, scope="tensor", stats=True,
                             workspace=ws)
    torch.cuda.synchronize()
    assert int(st.status.item()) == 0
    units = st.units_numpy()[0]
    # embedding, layer 0 (q, k, o, gate, down, norm), layer 27 (v, up)
    picks = [0, 1, 2, 4, 5, 7, 8, 1 + 27 * 9 + 2, 1 + 27 * 9 + 5]
    for q in picks:
        a, b = to_np(th0[q]), to_np(th1[q])
        r = oracle.update([a.reshape(shapes[q][0], shapes[q][1])], [b.reshape(shapes[q][0], shapes[q][1])],
                          oracle.ISO, update_is_delta=False, density=0.05, is_1d=[shapes[q][2]])
        assert_values_close(to_np(out[q]), r["out64"][0], r["mag"][0], f"full-size tensor {q}",
                            op="iso", K=1)
        assert_units_equal(units[q:q + 1], r["units"][0], f"full-size unit {q}")
        if shapes[q][2]:
            assert units[q]["k"] == -1      # 1-D tensors take the ISO average, untrimmed
    del th0, th1, out
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------
# the fused K = 1 pass: each way it falls back to the full exact apply
# ---------------------------------------------------------------------------
def _update_vs_oracle(th0, th1, op, density, is_delta=False, what=""):
    shapes = [(t.shape[0], t.shape[1]) if t.dim() == 2 else (1, t.numel()) for t in th0]
    is1d = [t.dim() == 1 for t in th0]
    out, st = iso.iso_update([t.to(DEV) for t in th0], [t.to(DEV) for t in th1], op=op,
                             update_is_delta=is_delta, density=density, stats=True)
    torch.cuda.synchronize()
    r = oracle.update(_np_list(th0), _np_list(th1), OPS[op], update_is_delta=is_delta,
                      density=density, shapes=shapes, is_1d=is1d)
    _check_merge(out, st, r, th0, OPS[op], 1, what=what)
    return r


def test_fused_repair_when_retention_coefficient_is_not_one():
    # ||trimmed tau||^2 ~ 1e-13 < 2^25 * ridge: c = Gamma / (Gamma + ridge) is far from 1
    g = torch.Generator().manual_seed(31)
    th0 = (torch.randn(300, 1000, generator=g) * 0.02).to(torch.bfloat16)
    tiny = (torch.randn(300, 1000, generator=g) * 1e-9)
    r = _update_vs_oracle([th0], [tiny], "iso", 0.05, is_delta=True, what="tiny-gamma iso")
    assert 0.0 < r["coef"][0][0] < 0.9


def test_fused_repair_when_band_records_overflow():
    # every |tau| equal: the whole tensor is one run of ties at the threshold
    g = torch.Generator().manual_seed(32)
    th0 = (torch.randn(300, 1000, generator=g) * 0.02).to(torch.bfloat16)
    sgn = torch.where(torch.rand(300, 1000, generator=g) < 0.5, -1.0, 1.0)
    d = (sgn * 2.0 ** -10).to(torch.bfloat16)
    for op in ("ties", "iso"):
        _update_vs_oracle([th0], [d], op, 0.05, is_delta=True, what=f"all-tied {op}")


def test_fused_bf16_delta_input_mixed_list():
    th0 = synth.base_weights(MIXED, seed=33)
    taus = [t.to(torch.bfloat16) for t in _taus(MIXED, 34, torch.float32)]
    for op in ("ties", "iso"):
        _update_vs_oracle(th0, taus, op, 0.05, is_delta=True, what=f"bf16 delta {op}")


LARGE_GLOBAL = [(4096, 8192, False), (1, 4096, True), (4096, 8192, False), (3000, 7001, False)]


@pytest.mark.parametrize("op,density", [("ties", 0.2), ("iso", 0.05), ("ties", 0.5)])
def test_global_unit_with_a_large_pool_and_many_tiles(op, density):
    # one GLOBAL unit of 88 M entries: more than 65536 tiles (the cut picks
    # its chunk from per-chunk tie sums first) and a band of candidates above
    # 2^20 keys (histogrammed as one flat pool, the count pass sealing the
    # unused slots of its chunks); bf16 checkpoints give long runs of ties
    th0, th1 = synth.rl_update_set(LARGE_GLOBAL, seed=43)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    out, st = iso.iso_update(d0, d1, op=op, update_is_delta=False, density=density, scope="global",
                             lam=1.0, stats=True)
    torch.cuda.synchronize()
    r = oracle.update(_np_list(th0), _np_list(th1), OPS[op], update_is_delta=False, density=density,
                      scope=oracle.SCOPE_GLOBAL, lam=1.0, shapes=_shapes(LARGE_GLOBAL), is_1d=_is1d(LARGE_GLOBAL))
    _check_merge(out, st, r, th0, OPS[op], 1, what=f"large global {op} {density}")
    u = st.units_numpy()[0, 0]
    if op == "ties":
        assert u["ties_at_thresh"] > u["ties_taken"] > 0     # the cut splits a run of ties
