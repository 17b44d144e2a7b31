"""What float32 arithmetic does to the method, measured with a plain float32 restatement.

tests/f32_restatement.py evaluates the layer with IEEE float32 operations only. These
checks pin it to the float64 oracle on small layers (it is the method, rounded), then
measure it on the large layer workloads against the bounds the GPU parity tests use:
every large layer misses the stated 1e-6 rms absolute term of dL/dX somewhere, and meets
the 1e-5 rms reading of tests/parity.py with room to spare. That is the evidence behind
the reading: the stated term is tighter than float32 evaluation of the method allows.
On long horizons with a slow somatic decay (T >= 256, beta >= 0.9) the restatement misses
even the stated V^s bound or the grad_x reading: the evidence behind the derived
allowances that tests/parity.py adds for those layers only.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2412_06355_gb300 import workloads
from paper_2412_06355_gb300.workloads import WORKLOADS

import f32_restatement as f32r


def measure(w, inp=None):
    """Worst error over bound of the float32 restatement against the oracle: V^s at the
    stated bound, dL/dX with absolute terms 1e-6 and 1e-5 rms, parameter gradients at the
    stated bound."""
    inp = inp or workloads.make_inputs(w, "cpu")
    chan, mrow = oracle.layer_channels(w.B, w.N, w.C, w.inner, w.mask_per_neuron)
    x = oracle.layer_x(w, inp["x"])
    s_o, v_o = oracle.forward_layer(w, inp)
    v_o, s_o = v_o.reshape(w.T, -1), s_o.reshape(w.T, -1)
    amb = np.abs(v_o - w.theta) < 1e-5
    first = np.where(amb.any(0), amb.argmax(0), w.T)
    gs = inp["gs"].clone().reshape(w.T, -1)
    gs[:, torch.from_numpy(first < w.T)] = 0
    ref = oracle.backward_layer(w, inp, gs=gs.reshape(w.T, w.B, w.N))
    r = f32r.run(w, x, inp, chan, mrow, oracle.to_f64(gs))
    t_idx = np.arange(w.T)[:, None]
    out = {"v": float((np.abs(r["v"] - v_o) / (1e-6 + 1e-5 * np.abs(v_o)))[t_idx <= first].max()),
           "spike_mismatch": int(((r["s"] != s_o) & (t_idx < first)).sum())}
    want = ref["gx"].reshape(w.T, -1, w.K)
    err = np.abs(r["gx"].astype(np.float64) - want)
    rms = np.sqrt(np.mean(want ** 2))
    rt = 2e-2 if w.dtype == "bf16" else 1e-4
    out["gx_1e-6"] = float((err / (rt * np.abs(want) + 1e-6 * rms)).max())
    out["gx_1e-5"] = float((err / (rt * np.abs(want) + 1e-5 * rms)).max())
    for k in ("galpha", "gxi", "gzeta", "gkappa"):
        e = np.abs(r[k] - ref[k])
        out[k] = float((e / (1e-4 * np.abs(ref[k]) + 1e-6 * np.sqrt(np.mean(ref[k] ** 2)))).max())
    return out


SMALL = [
    workloads.Workload("s1", T=6, B=3, N=4 * 64, K=4, G=1, C=4, inner=64, dtype="f32",
                       psi="mh", reset="hard", seed=3),
    workloads.Workload("s2", T=9, B=2, N=3 * 32, K=8, G=2, C=3, inner=32, dtype="f32",
                       psi="identity", reset="soft", mask_p=0.5, seed=4),
    workloads.Workload("s3", T=5, B=2, N=2 * 48, K=8, G=1, C=2, inner=48, dtype="bf16",
                       psi="mh", reset="soft", mask_p=0.6, mask_per_neuron=True, seed=5),
    workloads.Workload("s4", T=12, B=2, N=2 * 40, K=4, G=4, C=2, inner=40, dtype="f32",
                       psi="mh", reset="hard", detach_reset=True, beta=0.9, seed=6),
]


@pytest.mark.parametrize("w", SMALL, ids=lambda w: w.name)
def test_restatement_is_the_method_rounded(w):
    m = measure(w)
    assert m["spike_mismatch"] == 0
    assert m["v"] < 1.0 and m["gx_1e-5"] < 1.0, m
    for k in ("galpha", "gxi", "gzeta", "gkappa"):
        assert m[k] < 1.0, (k, m)


def test_restatement_catches_a_wrong_parameter():
    """The comparison can see a slip: a branch strength off by 1e-3 in the restatement only
    moves V^s far outside its bound."""
    w = SMALL[0]
    inp = workloads.make_inputs(w, "cpu")
    chan, mrow = oracle.layer_channels(w.B, w.N, w.C, w.inner, w.mask_per_neuron)
    kappa = inp["kappa"].clone()
    kappa[0, 0] += 1e-3
    r = f32r.run(w, oracle.layer_x(w, inp["x"]), dict(inp, kappa=kappa), chan, mrow,
                 oracle.to_f64(inp["gs"].reshape(w.T, -1)))
    _, v_o = oracle.forward_layer(w, inp)
    v_o = v_o.reshape(w.T, -1)
    assert (np.abs(r["v"] - v_o) / (1e-6 + 1e-5 * np.abs(v_o))).max() > 10.0


LARGE = [WORKLOADS["conv"].with_(B=2), WORKLOADS["event"].with_(B=1),
         WORKLOADS["token_dbg"].with_(B=2)]


@pytest.mark.parametrize("w", LARGE, ids=lambda w: w.name)
def test_float32_misses_the_stated_grad_x_term_and_meets_the_reading(w):
    m = measure(w)
    assert m["spike_mismatch"] == 0 and m["v"] < 1.0, m
    assert m["gx_1e-6"] > 1.0, m            # the stated 1e-6 rms: float32 evaluation misses it
    assert m["gx_1e-5"] < 0.75, m           # the reading: met with room to spare
    for k in ("galpha", "gxi", "gzeta", "gkappa"):
        assert m[k] < 1.0, (k, m)


def test_float32_misses_the_bounds_on_long_slow_horizons():
    """The long-horizon layers at beta = 0.95 that the parity tests check with the derived
    allowances: a T = 2048 layer with identity branches (grad_x beyond even the 1e-5 rms
    reading) and a T = 300 bfloat16 layer with a soft reset and the residual term (V^s
    beyond its stated bound where V^s is near zero)."""
    long_t = WORKLOADS["long_t"].with_(B=1, N=1024, C=1, psi="identity")
    m = measure(long_t)
    assert m["gx_1e-5"] > 1.0, m
    soft = workloads.Workload("tp1", T=300, B=4, N=64, K=1, G=1, C=2, inner=32, dtype="bf16",
                              psi="identity", reset="soft", theta=0.6, beta=0.95, x_mean=0.1,
                              x_density=0.3, residual=True, seed=1)
    m = measure(soft)
    assert m["v"] > 1.0, m
