"""The oracle's pins catch plausible mistakes.

Each case copies the oracle's C source, plants one mistake (a dropped term, a
wrong sign, a reversed tie order, a wrong rounding ...), compiles the copy and
runs the pin suite against it: the suite must fail.  Everything runs on the CPU.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "iso_oracle.c")

MUTATIONS = {
    "tie_order_reversed_sort": ("if (x->pos != y->pos) return (x->pos < y->pos) ? -1 : 1;",
                                "if (x->pos != y->pos) return (x->pos > y->pos) ? -1 : 1;"),
    "one_tie_too_many": ("else if (kp == t && taken < need)", "else if (kp == t && taken <= need)"),
    "signed_key": ("return f32_bits(t) & 0x7FFFFFFFu;", "return f32_bits(t);"),
    "k_truncates": ("double kk = floor(rho * (double)n + 0.5);", "double kk = floor(rho * (double)n);"),
    "ties_disagreeing_set": ("if (tt != 0.0f && sign_f(tt) == gamma)", "if (tt != 0.0f && sign_f(tt) != gamma)"),
    "ties_plain_mean": ("double merged = cnt ? acc / (double)cnt : 0.0;",
                        "double merged = cnt ? acc / (double)K : 0.0;"),
    "ties_untrimmed_election": ("float tt = kept(mask, i, p) ? tau32[i][p] : 0.0f;", "float tt = tau32[i][p];"),
    "ta_drops_lambda": ("out[p] = add_update(theta0[p], lambda * s);", "out[p] = add_update(theta0[p], s);"),
    "retention_rhs_ones": ("b[r] = gram[idx[r] * K + idx[r]];", "b[r] = 1.0;"),
    "retention_no_clip": ("if (c > c_max) c = c_max;", ";"),
    "gram_diagonal_only": ("s += gi * gj;", "s += gi * gi;"),
    "gram_untrimmed": ("double gi = kept(mask, i, p) ? tau64[i][p] : 0.0;", "double gi = tau64[i][p];"),
    "iso_1d_no_average": ("out[p] = add_update(theta0[p], s / (double)K);", "out[p] = add_update(theta0[p], s);"),
    "bf16_round_half_up": ("u += 0x7FFFu + lsb;", "u += 0x8000u;"),
    "bf16_f64_truncates": ("double q = round_half_even(ldexp(a, -q_exp));", "double q = floor(ldexp(a, -q_exp));"),
    "ram_threshold_inclusive": ("if (fabs((double)tau32[i][p]) > eps_act) active[c++] = i;",
                                "if (fabs((double)tau32[i][p]) >= eps_act) active[c++] = i;"),
    "ram_mean_over_all_experts": ("tau_ram = s / (double)c;", "tau_ram = s / (double)K;"),
    "ram_unique_value_divided": ("tau_ram = tau64[active[0]][p];", "tau_ram = tau64[active[0]][p] / (double)K;"),
    "ram_drops_lambda": ("out[p] = add_update(theta0[p], lambda * tau_ram);", "out[p] = add_update(theta0[p], tau_ram);"),
    "ram_inactive_kept": ("if (c == 0) {\n            tau_ram = 0.0;",
                          "if (c == 0) {\n            tau_ram = tau64[0][p];"),
    "zero_update_normalises_sign": ("return (upd == 0.0) ? theta0 : theta0 + upd;", "return theta0 + upd;"),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, tmp_path):
    old, new = MUTATIONS[name]
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation anchor not found: {name}"
    mdir = tmp_path / "oracle_mut"
    mdir.mkdir()
    shutil.copy(os.path.join(ROOT, "oracle", "iso_oracle.h"), mdir / "iso_oracle.h")
    (mdir / "iso_oracle.c").write_text(src.replace(old, new))
    so = mdir / "libmut.so"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fPIC", "-shared",
                           "-o", str(so), str(mdir / "iso_oracle.c"), "-lm"])
    env = dict(os.environ, ISO_ORACLE_LIB=str(so))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch mutation {name}:\n{r.stdout[-2000:]}"


# ---------------------------------------------------------------------------
# the frame-space ISO-Merger oracle (numpy): the same scheme on its source
# ---------------------------------------------------------------------------
MERGER_SRC = os.path.join(ROOT, "oracle", "iso_merger.py")
MERGER_MUTATIONS = {
    "sym_drops_half": ("return 0.5 * (A + A.T)", "return (A + A.T)"),
    "projection_skipped": ("return D - U0 @ sym(U0.T @ D)", "return D"),
    "sign_zero_negative": ("s[s == 0] = 1.0", "s[s == 0] = -1.0"),
    "no_sign_canonicalization": ("Ui, Vi, s = canonicalize_signs(U0, Ui, Vi)", "s = np.ones(Ui.shape[1])"),
    "mask_keeps_every_mode": ("out[:, k_keep:] = 0.0", "out[:, k_keep:] *= 1.0"),
    "k_keep_truncates": ("k = int(np.floor(rho_keep * q + 0.5))", "k = int(np.floor(rho_keep * q))"),
    "proxy_drops_v_motion": ("return (xiU * S0) @ V0.T + (U0 * S0) @ xiV.T", "return (xiU * S0) @ V0.T"),
    "aggregate_not_projected": ("return tangent_project(U0, agg)", "return agg"),
    "retraction_without_polar": ("return polar(U0 + xi)", "return U0 + xi"),
    "gram_diagonal_only": ("gram[i, j] = float(np.sum(g[i] * g[j]))", "gram[i, j] = float(np.sum(g[i] * g[i]))"),
    "coefficients_unused": ("agg += c[i] * xis[i]", "agg += xis[i]"),
}


@pytest.mark.parametrize("name", sorted(MERGER_MUTATIONS))
def test_merger_pins_catch_mutation(name, tmp_path):
    old, new = MERGER_MUTATIONS[name]
    src = open(MERGER_SRC).read()
    assert src.count(old) == 1, f"mutation anchor not found: {name}"
    src = src.replace("from . import retention as _retention", "from oracle import retention as _retention")
    path = tmp_path / "iso_merger_mut.py"
    path.write_text(src.replace(old, new))
    env = dict(os.environ, ISO_MERGER_PATH=str(path))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_iso_merger.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch mutation {name}:\n{r.stdout[-2000:]}"


# ---------------------------------------------------------------------------
# the ISO-Optimizer oracle (numpy): the same scheme on its source
# ---------------------------------------------------------------------------
OPT_SRC = os.path.join(ROOT, "oracle", "iso_optimizer.py")
OPT_MUTATIONS = {
    "grad_u_without_sigma": ("return (G_W @ V) * S0[None, :], (G_W.T @ U) * S0[None, :]",
                             "return (G_W @ V), (G_W.T @ U) * S0[None, :]"),
    "grad_v_from_v": ("(G_W.T @ U) * S0[None, :]", "(G_W.T @ U[:, ::-1]) * S0[None, :]"),
    "no_bias_correction": ("bc1 = 1.0 - beta1 ** step", "bc1 = 1.0"),
    "eps_inside_sqrt": ("np.sqrt(v / bc2) + eps", "np.sqrt(v / bc2 + eps)"),
    "coupled_decay": ("X - lr * weight_decay * X", "X - weight_decay * X"),
    "second_moment_of_abs": ("(1.0 - beta2) * g * g", "(1.0 - beta2) * np.abs(g)"),
    "no_retraction": ("    return P @ Qt", "    return np.asarray(X, np.float64)"),
}


@pytest.mark.parametrize("name", sorted(OPT_MUTATIONS))
def test_optimizer_pins_catch_mutation(name, tmp_path):
    old, new = OPT_MUTATIONS[name]
    src = open(OPT_SRC).read()
    assert src.count(old) == 1, f"mutation anchor not found: {name}"
    path = tmp_path / "iso_optimizer_mut.py"
    path.write_text(src.replace(old, new))
    env = dict(os.environ, ISO_OPTIMIZER_PATH=str(path))
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_iso_optimizer.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode != 0, f"pins did not catch mutation {name}:\n{r.stdout[-2000:]}"
