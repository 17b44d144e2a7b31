"""Pins of the float64 point-neuron LIF oracle (the DendSN soma driven by one current).

The LIF layer is the baseline the paper measures the DendSN layer's speed against
(Results, efficiency paragraph); its neuron is the soma of Eq. methods-lif-reset-charge
and Eq. methods-lif-fire with the input current in place of Z. Pins:

* the hand-derived worked trajectories of tests/golden (fed with their Z sequence);
* the geometric-series closed form below threshold and the resulting firing period;
* the closed-form gradient of a sub-threshold layer, dV[t]/dX[s] = beta^(t-s);
* central finite differences of the smooth-spike forward (Eq. methods-sg primitive);
* an independent float64 torch.autograd restatement with the surrogate spike;
* the DendSN oracle reduced to a point neuron (one compartment, identity psi,
  stateless, kappa = 1, xi = 0, zeta = 1, positive inputs, so Z = X exactly).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import LIFConfig, OracleConfig, backward, forward, lif_backward, lif_forward

HERE = os.path.dirname(os.path.abspath(__file__))


def test_lif_golden_worked_trajectories():
    cases = json.load(open(os.path.join(HERE, "golden", "lif_worked_trajectories.json")))["cases"]
    for c in cases:
        # the golden neuron's soma is driven by Z[t] = |V^d[t]| with V^d the leaky
        # compartment (one compartment, identity psi, kappa = 1, xi = 0, zeta = 1)
        z, vd = [], 0.0
        for xt in c["x"]:
            vd = c["alpha"] * vd + xt
            z.append(abs(vd))
        cfg = LIFConfig(T=len(z), reset=c["reset"], theta=c["theta"], beta=c["beta"])
        s, v = lif_forward(cfg, np.array(z)[:, None])
        assert v[:, 0].tolist() == c["v"], c["name"]
        assert s[:, 0].tolist() == c["s"], c["name"]


@pytest.mark.parametrize("c,beta", [(0.3, 0.5), (0.11, 0.9), (0.7, 0.0)])
def test_lif_constant_input_geometric_series_and_period(c, beta):
    T = 40
    theta = 1.0
    s, v = lif_forward(LIFConfig(T=T, theta=theta, beta=beta), np.full((T, 1), c))
    # before the first spike V[t] = c (1 - beta^(t+1)) / (1 - beta); after a hard
    # reset the trajectory restarts from V = c, so the spike train is periodic
    closed = [c * (1 - beta ** (t + 1)) / (1 - beta) for t in range(T)]
    first = next((t for t in range(T) if closed[t] >= theta), None)
    if first is None:
        np.testing.assert_allclose(v[:, 0], closed, rtol=1e-14)
        assert s.sum() == 0
        return
    period = first + 1
    for t in range(T):
        np.testing.assert_allclose(v[t, 0], closed[t % period], rtol=1e-14)
        assert s[t, 0] == (1.0 if t % period == first else 0.0)


# (the soft reset's path carries sg(V - theta) * beta * theta, about 7e-11 at
# theta = 1e9: not zero, so the soft case detaches it to make the closed form exact)
@pytest.mark.parametrize("reset,detach", [("hard", False), ("hard", True), ("soft", True)])
def test_lif_subthreshold_gradient_closed_form(reset, detach):
    rng = np.random.default_rng(3)
    T, M, beta = 9, 5, 0.7
    x = rng.normal(0.0, 0.2, (T, M))
    gv = rng.normal(size=(T, M))
    cfg = LIFConfig(T=T, reset=reset, theta=1e9, beta=beta, detach_reset=detach)  # never fires
    gx = lif_backward(cfg, x, np.zeros((T, M)), gv)
    want = np.zeros((T, M))
    for s_ in range(T):
        for t in range(s_, T):
            want[s_] += gv[t] * beta ** (t - s_)
    np.testing.assert_allclose(gx, want, rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("reset,detach", [("hard", False), ("soft", False), ("hard", True)])
def test_lif_smooth_spike_finite_differences(reset, detach):
    rng = np.random.default_rng(5)
    T, M = 6, 3
    x = rng.normal(0.6, 0.5, (T, M))
    ws, wv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    cfg = LIFConfig(T=T, reset=reset, theta=1.0, beta=0.6, smooth_spike=True,
                    detach_reset=detach)
    gx = lif_backward(cfg, x, ws, wv)
    if detach:
        # a detached reset path is not the derivative of this forward (the autograd
        # restatement below checks it); here only: it does change the gradient
        full = lif_backward(LIFConfig(T=T, reset=reset, theta=1.0, beta=0.6, smooth_spike=True),
                            x, ws, wv)
        assert np.abs(full - gx).max() > 1e-6
        return

    def loss(x_):
        s, v = lif_forward(cfg, x_)
        return float((ws * s).sum() + (wv * v).sum())

    h = 1e-5
    fd = np.zeros_like(x)
    for idx in np.ndindex(*x.shape):
        xp, xm = x.copy(), x.copy()
        xp[idx] += h
        xm[idx] -= h
        fd[idx] = (loss(xp) - loss(xm)) / (2 * h)
    np.testing.assert_allclose(gx, fd, rtol=1e-6, atol=1e-8)


class _Spike(torch.autograd.Function):
    """Heaviside forward (Theta(0) = 1), arctan-surrogate backward (Eq. methods-sg)."""

    @staticmethod
    def forward(ctx, u):
        ctx.save_for_backward(u)
        return (u >= 0).to(u.dtype)

    @staticmethod
    def backward(ctx, g):
        (u,) = ctx.saved_tensors
        return g / (1 + (math.pi * u) ** 2)


def torch_lif(x, reset, theta, beta, detach):
    v = torch.zeros_like(x[0])
    s = torch.zeros_like(x[0])
    vs, ss = [], []
    for t in range(x.shape[0]):
        sr = s.detach() if detach else s
        if reset == "hard":
            v = beta * (1 - sr) * v + x[t]
        else:
            v = beta * (v - theta * sr) + x[t]
        s = _Spike.apply(v - theta)
        vs.append(v)
        ss.append(s)
    return torch.stack(ss), torch.stack(vs)


LIF_AUTOGRAD = [("hard", False, 1.0), ("soft", False, 1.0), ("hard", True, 1.0),
                ("soft", True, 1.0), ("soft", False, 0.75), ("hard", False, 0.75)]


@pytest.mark.parametrize("reset,detach,theta", LIF_AUTOGRAD)
def test_lif_backward_matches_autograd_restatement(reset, detach, theta):
    rng = np.random.default_rng(8)
    T, M = 12, 40
    x = rng.normal(0.5 * theta, 0.6, (T, M))
    gs, gv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    cfg = LIFConfig(T=T, reset=reset, theta=theta, beta=0.5, detach_reset=detach)
    s_o, v_o = lif_forward(cfg, x)
    xt = torch.tensor(x, requires_grad=True)
    s_t, v_t = torch_lif(xt, reset, theta, 0.5, detach)
    assert np.array_equal(s_t.detach().numpy(), s_o)
    np.testing.assert_allclose(v_t.detach().numpy(), v_o, rtol=1e-14, atol=1e-15)
    ((s_t * torch.tensor(gs)).sum() + (v_t * torch.tensor(gv)).sum()).backward()
    gx = lif_backward(cfg, x, gs, gv)
    np.testing.assert_allclose(gx, xt.grad.numpy(), rtol=1e-12, atol=1e-13)
    assert s_o.sum() > 0                 # the case does exercise the reset


@pytest.mark.parametrize("reset", ["hard", "soft"])
def test_lif_is_the_dendsn_reduced_to_a_point_neuron(reset):
    rng = np.random.default_rng(9)
    T, M = 10, 30
    x = np.abs(rng.normal(0.5, 0.6, (T, M))) + 1e-3          # Z = |X| = X
    gs, gv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    lc = LIFConfig(T=T, reset=reset, theta=1.0, beta=0.5)
    dc = OracleConfig(T=T, K=1, G=1, C=1, psi="identity", reset=reset, stateless=True)
    one = [np.zeros((1, 1)), np.zeros((1, 1)), np.ones((1, 1)), np.ones((1, 1))]
    chan = np.zeros(M, np.int32)
    s_l, v_l = lif_forward(lc, x)
    s_d, v_d = forward(dc, x[:, :, None], chan, None, *one)
    assert np.array_equal(s_l, s_d) and np.array_equal(v_l, v_d)
    g_l = lif_backward(lc, x, gs, gv)
    g_d = backward(dc, x[:, :, None], chan, None, *one, None, gs, gv)["gx"][:, :, 0]
    np.testing.assert_allclose(g_l, g_d, rtol=1e-13, atol=1e-15)
