"""GPU parity of the fused single-pass K = 1 update.

The fused pass writes speculative outputs from the sampled threshold and
corrects them exactly afterwards.  Each case is checked against the oracle and
against the library's two-pass form (which must give identical bits), and the
cases are built so that every correction path runs: the tie-run mode with the
sampled cut far from the exact one, a tie-run guess that misses the
threshold (full re-apply), the band mode with several key values, and the
exact sample of small tensors.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_19331_gb300 as iso
import synth
from paper_2607_19331_gb300 import _abi
from parity_util import assert_units_equal, assert_values_close, to_np

pytestmark = pytest.mark.gpu
DEV = "cuda:0"
OPS = {"ties": oracle.TIES, "iso": oracle.ISO}
S, C = 24576, 256          # the library's sample size and chunk length


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    torch.cuda.set_device(0)
    _abi.lib()
    yield
    iso.force_two_pass(False)


def sample_chunk_starts(n):
    nch = S // C
    return [0 if c == 0 else (int((n - C) * c / (nch - 1)) & ~7) for c in range(nch)]


def _run(th0, th1, op, density, is_delta, two_pass):
    iso.force_two_pass(two_pass)
    try:
        out, st = iso.iso_update([t.to(DEV) for t in th0], [t.to(DEV) for t in th1], op=op,
                                 update_is_delta=is_delta, density=density, stats=True)
        torch.cuda.synchronize()
    finally:
        iso.force_two_pass(False)
    assert int(st.status.item()) == 0
    return out, st


def check_fused(th0, th1, op, density, is_delta=False, what=""):
    """Fused vs oracle (values, units, coefficients) and fused vs two-pass (bits)."""
    out_f, st_f = _run(th0, th1, op, density, is_delta, False)
    out_t, st_t = _run(th0, th1, op, density, is_delta, True)
    shapes = [(t.shape[0], t.shape[1]) if t.dim() == 2 else (1, t.numel()) for t in th0]
    is1d = [t.dim() == 1 for t in th0]
    r = oracle.update([to_np(t) for t in th0], [to_np(t) for t in th1], OPS[op],
                      update_is_delta=is_delta, density=density, shapes=shapes, is_1d=is1d)
    for q in range(len(th0)):
        assert_values_close(to_np(out_f[q]), r["out64"][q], r["mag"][q], f"{what} fused tensor {q}",
                            op=op, K=1)
        assert np.array_equal(to_np(out_f[q]), to_np(out_t[q])), f"{what}: fused and two-pass differ, tensor {q}"
    uf = st_f.units_numpy()
    assert_units_equal(uf, r["units"], what)
    assert_units_equal(uf, st_t.units_numpy(), what + " (two-pass)")
    if op == "iso":
        cf = st_f.coef.cpu().numpy()[: len(th0)]
        np.testing.assert_array_equal(cf, st_t.coef.cpu().numpy()[: len(th0)])
        np.testing.assert_allclose(cf, np.array([c[0] for c in r["coef"]]), rtol=1e-5, atol=1e-9)
    return uf


@pytest.mark.parametrize("op", ["iso", "ties"])
@pytest.mark.parametrize("density", [0.05, 0.2])
def test_fused_qwen_shaped_checkpoints(op, density):
    shapes = synth.qwen_shapes("qwen1.5b", layers=2, scale=4)
    th0, th1 = synth.rl_update_set(shapes, seed=5)
    check_fused(th0, th1, op, density, what=f"qwen/4 {op} {density}")


def test_fused_small_and_ragged_tensors_take_the_exact_sample():
    shapes = [(300, 1000, False), (257, 129, False), (1, 1536, True), (3, 7, False), (0, 5, False),
              (64, 300, False), (1, 5, True), (40, 1000, False)]
    th0, th1 = synth.rl_update_set(shapes, seed=6)
    for op in ("iso", "ties"):
        check_fused(th0, th1, op, 0.05, what=f"mixed {op}")


def _tie_case(n_rows=400, n_cols=1000, seed=7, extra_ties_in_gaps=0, sampled_value=None):
    """bf16 task vector with three magnitudes: 'above' entries, a run of ties
    at v = 2^-10, and small background values, plus optional extra ties placed
    only between the sampled chunks (which the sample cannot see)."""
    n = n_rows * n_cols
    g = torch.Generator().manual_seed(seed)
    x = (torch.rand(n, generator=g) * 2.0 ** -12)                  # background, below v
    perm = torch.randperm(n, generator=g)
    x[perm[:30000]] = 2.0 ** -8                                      # above v
    x[perm[30000:60000]] = 2.0 ** -10                                # the tie run
    if extra_ties_in_gaps:
        starts = sample_chunk_starts(n)
        sampled = torch.zeros(n, dtype=torch.bool)
        for s0 in starts:
            sampled[s0:s0 + C] = True
        first_third = torch.arange(n) < n // 3
        cand = torch.nonzero(~sampled & first_third & (x < 2.0 ** -10)).flatten()
        pick = cand[torch.randperm(cand.numel(), generator=g)[:extra_ties_in_gaps]]
        x[pick] = 2.0 ** -10
    if sampled_value is not None:
        for s0 in sample_chunk_starts(n):
            x[s0:s0 + C] = sampled_value
    sgn = torch.where(torch.rand(n, generator=g) < 0.5, -1.0, 1.0)
    tau = (x * sgn).to(torch.bfloat16).reshape(n_rows, n_cols)
    th0 = (torch.randn(n_rows, n_cols, generator=g) * 0.02).to(torch.bfloat16)
    return th0, tau


def test_fused_tie_run_with_the_sampled_cut_far_from_the_exact_one():
    # 20000 extra ties hidden between the sampled chunks of the first third:
    # the sample places the cut near n/3, the exact cut is near n/9, and the
    # range between them is re-applied exactly
    th0, tau = _tie_case(extra_ties_in_gaps=20000)
    for op in ("ties", "iso"):
        u = check_fused([th0], [tau], op, 0.1, is_delta=True, what=f"hidden ties {op}")
        assert u[0, 0]["thresh_key"] == np.float32(2.0 ** -10).view(np.uint32)
        assert 0 < u[0, 0]["ties_taken"] < u[0, 0]["ties_at_thresh"]


def test_fused_tie_run_guess_that_misses_the_threshold():
    # every sampled entry holds the same value, so the sample proposes that
    # value as the threshold; the counts reject it and the tensor is
    # re-applied in full with the exact threshold
    th0, tau = _tie_case(sampled_value=2.0 ** -11)
    u = check_fused([th0], [tau], "ties", 0.1, is_delta=True, what="missed run")
    assert u[0, 0]["flags"] & 1, "expected the full-data fallback"


def test_fused_band_mode_with_several_key_values():
    # bf16(N(0, 1)): about 0.2 % of the entries share any one value near the
    # 10 % threshold, so the sampled band spans several values (band mode)
    g = torch.Generator().manual_seed(8)
    tau = torch.randn(512, 3000, generator=g).to(torch.bfloat16)
    th0 = (torch.randn(512, 3000, generator=g) * 0.02).to(torch.bfloat16)
    for op in ("ties", "iso"):
        check_fused([th0], [tau], op, 0.1, is_delta=True, what=f"band mode {op}")


def test_fused_checkpoint_update_in_place_matches():
    # an output aliasing theta_0 takes the two-pass form; the result is the same
    shapes = synth.qwen_shapes("qwen1.5b", layers=1, scale=8)
    th0, th1 = synth.rl_update_set(shapes, seed=9)
    d0, d1 = [t.to(DEV) for t in th0], [t.to(DEV) for t in th1]
    ref = iso.iso_update(d0, d1, op="iso", density=0.05)
    work = [t.clone() for t in d0]
    iso.iso_update(work, d1, op="iso", density=0.05, out=work)
    torch.cuda.synchronize()
    for a, b in zip(ref, work):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))
