"""Randomised parity sweep: layer configurations drawn from a fixed seed, each compared with
the float64 oracle element by element (tests/parity.py: tolerances, ambiguous steps, both
backward kernel builds).

Every knob of the ABI is drawn independently: K and G, channel count and width (including
widths that are and are not multiples of 32, so both paper-layout forwards run), T across
the chunk and checkpoint boundaries, batch, dtype, psi, reset, detached reset, Stateless and
residual dendrites, per-channel and per-neuron masks, layout, threshold and decay. The point-
neuron LIF layer gets the same treatment. Sizes stay where the oracle finishes in well under
a second per case.
"""
import random

import numpy as np
import pytest
import torch

import oracle
from paper_2412_06355_gb300 import binding, workloads

from parity import (BF16_ATOL_REL, BF16_RTOL, G_ATOL_REL, G_RTOL, V_ATOL, V_RTOL,
                    assert_close, check_layer, first_ambiguous_step)

pytestmark = pytest.mark.gpu

KG = [(1, 1), (2, 1), (2, 2), (4, 1), (4, 2), (4, 4), (8, 1), (8, 2), (8, 4),
      (16, 1), (16, 2), (16, 4)]


def draw_layer(i: int) -> workloads.Workload:
    r = random.Random(1000 + i)
    K, G = r.choice(KG)
    inner = r.choice([1, 3, 7, 32, 40, 64, 96, 256])
    C = r.choice([1, 2, 3, 5, 8])
    per_sample = C * inner
    reps = max(1, r.choice([1, 2, 3]) * (64 // per_sample if per_sample < 64 else 1))
    N = per_sample * reps
    T = r.choice([1, 2, 3, 4, 5, 8, 9, 12, 17, 33])
    B = r.choice([1, 2, 3])
    mask_p = r.choice([None, None, 0.5, 0.8])
    return workloads.Workload(
        f"fuzz{i}", T=T, B=B, N=N, K=K, G=G, C=C, inner=inner,
        dtype=r.choice(["f32", "f32", "bf16"]), psi=r.choice(["mh", "identity"]),
        reset=r.choice(["hard", "soft"]), theta=r.choice([1.0, 1.0, 0.6]),
        beta=r.choice([0.5, 0.5, 0.9, 0.0]), x_mean=r.choice([0.3, 0.6]),
        x_density=r.choice([1.0, 1.0, 0.3]), mask_p=mask_p,
        mask_per_neuron=bool(mask_p is not None and r.random() < 0.5),
        stateless=r.random() < 0.25, residual=r.random() < 0.25,
        detach_reset=r.random() < 0.2, layout=r.choice(["kinner", "paper"]), seed=i)


LAYERS = [draw_layer(i) for i in range(160)]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("these tests need a CUDA device")
    binding.load()
    oracle.build()


def _id(w):
    return (f"K{w.K}G{w.G}C{w.C}i{w.inner}T{w.T}B{w.B}-{w.dtype}-{w.psi}-{w.reset}"
            f"{'-sl' if w.stateless else ''}{'-res' if w.residual else ''}"
            f"{'-det' if w.detach_reset else ''}{'-m' if w.mask_p is not None else ''}"
            f"{'n' if w.mask_per_neuron else ''}-{w.layout}")


@pytest.mark.parametrize("w", LAYERS, ids=[_id(w) for w in LAYERS])
def test_random_layer(w):
    check_layer(w)


def draw_lif(i: int):
    r = random.Random(5000 + i)
    return dict(T=r.choice([1, 3, 4, 5, 8, 9, 16, 23]), B=r.choice([1, 2, 5]),
                N=r.choice([4, 7, 64, 333, 1024]), dtype=r.choice(["f32", "bf16"]),
                reset=r.choice(["hard", "soft"]), theta=r.choice([1.0, 0.7]),
                beta=r.choice([0.5, 0.9, 0.0]), detach=r.random() < 0.3, seed=i)


LIFS = [draw_lif(i) for i in range(48)]


@pytest.mark.parametrize("c", LIFS, ids=lambda c: "-".join(f"{k}{v}" for k, v in c.items()))
def test_random_lif(c):
    T, B, N = c["T"], c["B"], c["N"]
    inp = workloads.make_lif_inputs(T, B, N, c["dtype"], c["seed"], with_gv=True)
    oc = oracle.LIFConfig(T=T, reset=c["reset"], theta=c["theta"], beta=c["beta"],
                          detach_reset=c["detach"])
    s_o, v_o = oracle.lif_forward(oc, inp["x"])
    first = first_ambiguous_step(v_o, c["theta"])
    amb = torch.from_numpy(first < T)
    gs, gv = inp["gs"].clone(), inp["gv"].clone()
    gs[:, amb] = 0
    gv[:, amb] = 0
    cfg = binding.make_lif_config(T, B, N, c["dtype"], c["reset"], c["theta"], c["beta"],
                                  c["detach"])
    saved = binding.lif_workspace(cfg)
    x = inp["x"].cuda()
    s, v = binding.lif_forward(cfg, x, want_v=True, saved=saved)
    gx = binding.lif_backward(cfg, x, gs.cuda(), gv.cuda(), saved)
    torch.cuda.synchronize()
    t_idx = np.arange(T)[:, None, None]
    assert_close("V", oracle.to_f64(v), v_o, V_RTOL, 0.0, mask=t_idx <= first[None],
                 atol_abs=V_ATOL)
    sm = t_idx < first[None]
    assert np.array_equal(oracle.to_f64(s)[sm], s_o[sm])
    rt, ar = (BF16_RTOL, BF16_ATOL_REL) if c["dtype"] == "bf16" else (G_RTOL, G_ATOL_REL)
    assert_close("grad_x", oracle.to_f64(gx), oracle.lif_backward(oc, inp["x"], gs, gv), rt, ar)


# Layers that take the time-parallel kernels (at least 256 steps, at most 2048 neurons): the
# compartment scans run in parallel over time there, so every flag is exercised again.
def draw_tp_layer(i: int) -> workloads.Workload:
    r = random.Random(9000 + i)
    K, G = r.choice(KG)
    inner = r.choice([1, 7, 32, 64])
    C = r.choice([1, 2, 3])
    per_sample = C * inner
    N = per_sample * r.choice([1, 2])
    B = r.choice([1, 2, 4])
    T = r.choice([256, 257, 300, 640, 1000])
    mask_p = r.choice([None, 0.5])
    return workloads.Workload(
        f"tp{i}", T=T, B=B, N=N, K=K, G=G, C=C, inner=inner,
        dtype=r.choice(["f32", "f32", "bf16"]), psi=r.choice(["mh", "identity"]),
        reset=r.choice(["hard", "soft"]), theta=r.choice([1.0, 0.6]),
        beta=r.choice([0.5, 0.9, 0.95]), x_mean=r.choice([0.1, 0.3]),
        x_density=r.choice([1.0, 0.3]), mask_p=mask_p,
        mask_per_neuron=bool(mask_p is not None and r.random() < 0.5),
        stateless=r.random() < 0.25, residual=r.random() < 0.25,
        detach_reset=r.random() < 0.2, layout=r.choice(["kinner", "paper"]), seed=i)


TP_LAYERS = [draw_tp_layer(i) for i in range(40)]


@pytest.mark.parametrize("w", TP_LAYERS, ids=[_id(w) for w in TP_LAYERS])
def test_random_time_parallel_layer(w):
    assert binding.dendsn_workspace_size(binding.config_of(w))[0] == 0   # no checkpoints
    check_layer(w)


@pytest.mark.parametrize("reset", ["hard", "soft"])
@pytest.mark.parametrize("theta", [0.0, -0.3])
def test_time_parallel_nonpositive_threshold(reset, theta):
    """theta <= 0: V^s[-1] = 0 already reaches the threshold, yet no spike precedes step 0."""
    w = workloads.Workload("tp_theta", T=300, B=2, N=64, K=4, G=2, C=2, inner=32, dtype="f32",
                           psi="mh", reset=reset, theta=theta, beta=0.8, seed=77)
    assert binding.dendsn_workspace_size(binding.config_of(w))[0] == 0   # the time-parallel path
    check_layer(w)
