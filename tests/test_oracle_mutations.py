"""The oracle's pins must catch plausible mistakes in the oracle itself.

Each mutation below plants one slip in a copy of oracle/dendsn_oracle.c (a dropped term,
a flipped sign, a transposed operand, an off-by-one in time, a wrong constant), builds
it with gcc, and runs the pin tests against it: at least one pin must fail. This is the
evidence that the pins constrain every equation of the method, not just some.
"""
import os
import subprocess
import tempfile

import pytest

import oracle
import oracle.oracle as oracle_mod
import test_oracle_lif_pins as lif_pins
import test_oracle_pins as pins

# (id, text in the oracle source, replacement)
MUTATIONS = [
    ("scan_transposed", "alpha[i] * vd_prev[i] + xt[i]", "alpha[i] * xt[i] + vd_prev[i]"),
    ("scan_no_leak", "alpha[i] * vd_prev[i] + xt[i]", "vd_prev[i] + xt[i]"),
    ("affine_sign", "double u = (vd[i] - xi[i]) / zeta[b];", "double u = (vd[i] + xi[i]) / zeta[b];"),
    ("affine_mul", "double u = (vd[i] - xi[i]) / zeta[b];", "double u = (vd[i] - xi[i]) * zeta[b];"),
    ("norm_no_sqrt", "double r = sqrt(sq);", "double r = sq;"),
    ("mexhat_exponent", "return (1.0 - r * r) * exp(-0.5 * r * r);", "return (1.0 - r * r) * exp(-r * r);"),
    ("mexhat_deriv", "return r * (r * r - 3.0) * exp(-0.5 * r * r);", "return r * (r * r - 1.0) * exp(-0.5 * r * r);"),
    ("hard_reset_dropped", "v = cfg->beta * (1.0 - s_prev) * v_prev + z;", "v = cfg->beta * v_prev + z;"),
    ("soft_reset_theta", "v = cfg->beta * (v_prev - cfg->theta * s_prev) + z;", "v = cfg->beta * (v_prev - s_prev) + z;"),
    ("heaviside_strict", "return (v - cfg->theta >= 0.0) ? 1.0 : 0.0;", "return (v - cfg->theta > 0.0) ? 1.0 : 0.0;"),
    ("surrogate_pi", "return 1.0 / (1.0 + ORACLE_PI * ORACLE_PI * x * x);", "return 1.0 / (1.0 + ORACLE_PI * x * x);"),
    ("reset_grad_sign", "dvds_next = -cfg->beta * vs[t];", "dvds_next = cfg->beta * vs[t];"),
    ("reset_gate_grad", "dvdv_next = cfg->beta * (1.0 - s[t]);", "dvdv_next = cfg->beta;"),
    ("soft_reset_grad", "dvds_next = -cfg->beta * cfg->theta;", "dvds_next = -cfg->beta;"),
    ("zeta_grad_sign", "gzeta[(int64_t)ch * Kb + b] -= dr * r / z_[b];", "gzeta[(int64_t)ch * Kb + b] += dr * r / z_[b];"),
    ("kappa_grad_mask", "gkappa[(int64_t)ch * Kb + b] += mk[b] * y * dz;", "gkappa[(int64_t)ch * Kb + b] += y * dz;"),
    ("scan_grad_dropped", "A[i] = direct[i] + a[i] * A[i];", "A[i] = direct[i];"),
    ("alpha_grad_time", "const double *vd_prev = vd_hist + (int64_t)t * K;\n            for (int i = 0; i < K; ++i) {\n                A[i]",
     "const double *vd_prev = vd_hist + (int64_t)(t + 1) * K;\n            for (int i = 0; i < K; ++i) {\n                A[i]"),
    ("xi_grad_sign", "gxi[(int64_t)ch * K + i] -= direct[i];", "gxi[(int64_t)ch * K + i] += direct[i];"),
    ("residual_mean", "z += mean / K;", "z += mean;"),
    ("mask_ignored", "km[b] = kappa[(int64_t)ch * Kb + b] * mb;", "km[b] = kappa[(int64_t)ch * Kb + b];"),
    ("direct_no_zeta", "direct[i] = du / z_[b];", "direct[i] = du;"),
    ("gv_dropped", "dv += gv[(int64_t)t * M + m];", "dv += 0.0;"),
    ("residual_grad", "g += dz / K;", "g += dz;"),
    # the learnable somatic decay (PLIF soma)
    ("gbeta_hard_leak", "(1.0 - s[t]) * vs[t] : vs[t] - cfg->theta * s[t];",
     "vs[t] : vs[t] - cfg->theta * s[t];"),
    ("gbeta_soft_theta", "(1.0 - s[t]) * vs[t] : vs[t] - cfg->theta * s[t];",
     "(1.0 - s[t]) * vs[t] : vs[t] - s[t];"),
    ("gbeta_wrong_step", "gbeta[ch] += dv_next * leak;", "gbeta[ch] += gs[(int64_t)t * M + m] * leak;"),
    # the point-neuron LIF layer
    ("lif_reset_dropped", "v = cfg->beta * (1.0 - s) * v + xt;", "v = cfg->beta * v + xt;"),
    ("lif_soft_theta", "v = cfg->beta * (v - cfg->theta * s) + xt;", "v = cfg->beta * (v - s) + xt;"),
    ("lif_bwd_recompute_reset", "vv = cfg->beta * (1.0 - ss) * vv + in;", "vv = cfg->beta * vv + in;"),
    ("lif_bwd_reset_gate", "a_vv = cfg->beta * (1.0 - st[t]);", "a_vv = cfg->beta;"),
    ("lif_bwd_reset_sign", "a_vs = -cfg->beta * vt[t];", "a_vs = cfg->beta * vt[t];"),
    ("lif_bwd_soft_theta", "a_vs = -cfg->beta * cfg->theta;", "a_vs = -cfg->beta;"),
    ("lif_bwd_gv_dropped", "g_v += gv[(int64_t)t * M + m];", "g_v += 0.0;"),
    ("lif_bwd_no_carry", "g_next = g_v;", "g_next = 0.0;"),
]

PIN_TESTS = [
    pins.test_golden_worked_trajectories,
    pins.test_constant_input_double_geometric_series,
    pins.test_plain_lif_firing_period,
    pins.test_soft_reset_unrolled_sum,
    pins.test_mexican_hat_is_minus_gaussian_second_derivative,
    pins.test_mexican_hat_derivative_roots,
    pins.test_l2_branch_aggregation_pythagorean,
    pins.test_arctan_surrogate_values,
    pins.test_kappa_linearity_and_mask_equals_zero_strength,
    pins.test_residual_with_zero_strength_is_lif_on_mean_input,
    lambda: pins.test_backward_matches_finite_differences(pins.VARIANTS[4], "smooth_spike"),
    lambda: pins.test_backward_matches_finite_differences(pins.VARIANTS[7], "subthreshold"),
    lambda: pins.test_backward_matches_autograd_restatement(pins.VARIANTS[3]),
    lambda: pins.test_backward_matches_autograd_restatement(pins.VARIANTS[1]),
    lambda: pins.test_backward_matches_autograd_restatement(pins.VARIANTS[7]),
    lif_pins.test_lif_golden_worked_trajectories,
    lambda: lif_pins.test_lif_constant_input_geometric_series_and_period(0.3, 0.5),
    lambda: lif_pins.test_lif_subthreshold_gradient_closed_form("hard", False),
    lambda: lif_pins.test_lif_smooth_spike_finite_differences("hard", False),
    lambda: lif_pins.test_lif_smooth_spike_finite_differences("soft", False),
    *[(lambda a=a: lif_pins.test_lif_backward_matches_autograd_restatement(*a))
      for a in lif_pins.LIF_AUTOGRAD],
]


def build_mutant(src: str, find: str, repl: str, out_dir: str, name: str) -> str:
    assert src.count(find) == 1, f"mutation anchor for {name} must occur exactly once"
    c = os.path.join(out_dir, name + ".c")
    so = os.path.join(out_dir, name + ".so")
    with open(c, "w") as f:
        f.write(src.replace(find, repl))
    subprocess.check_call(["gcc", "-O2", "-std=c99", "-ffp-contract=off", "-shared", "-fPIC",
                           c, "-o", so, "-lm"])
    return so


def caught(so_path: str) -> list:
    failures = []
    with oracle_mod.using_library(so_path):
        for i, t in enumerate(PIN_TESTS):
            try:
                t()
            except (AssertionError, RuntimeError, ValueError, FloatingPointError):
                failures.append(i)
    return failures


def test_unmutated_oracle_passes_the_selected_pins():
    oracle.build()
    for t in PIN_TESTS:
        t()


@pytest.mark.parametrize("name,find,repl", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_pins_catch_mutation(name, find, repl, tmp_path):
    src = open(oracle_mod.source_path()).read()
    so = build_mutant(src, find, repl, str(tmp_path), name)
    failed = caught(so)
    assert failed, f"no pin caught the mutation {name}"
