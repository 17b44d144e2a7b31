"""Pins of the float64 oracle against facts fixed by the paper and by mathematics.

Each pin is chosen so that a plausible slip in the oracle (a dropped term, a
wrong sign or index, a transposed operand) breaks at least one of them:

* hand-derived worked trajectories (tests/golden/lif_worked_trajectories.json)
* closed forms: geometric-series membrane trajectories, the plain-LIF period
* the Mexican hat as minus the second derivative of a Gaussian (Supplementary
  "Dendritic branch activation functions"), its roots and value at 0
* Pythagorean L2 branch aggregation (Eq. methods-branch-aggregation)
* the arctan surrogate's values (Eq. methods-sg)
* finite differences of the potential path and of a smooth-spike forward
* an independent float64 torch.autograd restatement of the forward, whose
  automatic gradient must equal the oracle's hand-derived backward
* invariants: kappa linearity, masking == zero strength, K identical branches,
  stateless == stateful with alpha = 0, per-channel parameter-gradient sums
"""
import dataclasses
import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import OracleConfig, forward, backward, layer_channels

HERE = os.path.dirname(os.path.abspath(__file__))


def one_neuron_params(K, Kb, alpha=0.0, xi=0.0, zeta=1.0, kappa=1.0, C=1):
    return (np.full((C, K), alpha), np.full((C, K), xi), np.full((C, Kb), zeta),
            np.full((C, Kb), kappa))


def run1(cfg, xs, **params):
    """Forward of one neuron per column of xs ([T, M, K])."""
    xs = np.asarray(xs, np.float64)
    M = xs.shape[1]
    a, xi, z, k = one_neuron_params(cfg.K, cfg.Kb, **params)
    return forward(cfg, xs, np.zeros(M, np.int32), None, a, xi, z, k)


# --------------------------------------------------------------------------- golden
def test_golden_worked_trajectories():
    with open(os.path.join(HERE, "golden", "lif_worked_trajectories.json")) as f:
        gold = json.load(f)
    for case in gold["cases"]:
        T = len(case["x"])
        cfg = OracleConfig(T=T, K=1, G=1, C=1, psi="identity", reset=case["reset"],
                           theta=case["theta"], beta=case["beta"])
        x = np.array(case["x"], np.float64).reshape(T, 1, 1)
        s, v = run1(cfg, x, alpha=case["alpha"])
        assert np.array_equal(v[:, 0], np.array(case["v"])), case["name"]
        assert np.array_equal(s[:, 0], np.array(case["s"], np.float64)), case["name"]


# --------------------------------------------------------------------------- closed forms
def test_constant_input_double_geometric_series():
    """No spikes: V^d[t] = c(1-a^t)/(1-a); V^s[t] = c/(1-a)[(1-b^t)/(1-b) - a(a^t-b^t)/(a-b)]."""
    T, c, a, b = 16, 0.3, 0.8, 0.5
    cfg = OracleConfig(T=T, K=1, G=1, C=1, psi="identity", reset="hard", theta=1e9, beta=b)
    s, v = run1(cfg, np.full((T, 1, 1), c), alpha=a)
    t = np.arange(1, T + 1, dtype=np.float64)
    want = c / (1 - a) * ((1 - b ** t) / (1 - b) - a * (a ** t - b ** t) / (a - b))
    np.testing.assert_allclose(v[:, 0], want, rtol=1e-13, atol=0)
    assert not s.any()
    # alpha = 0: V^s[t] = c(1-b^t)/(1-b)
    s, v = run1(cfg, np.full((T, 1, 1), c), alpha=0.0)
    np.testing.assert_allclose(v[:, 0], c * (1 - b ** t) / (1 - b), rtol=1e-13)


def test_plain_lif_firing_period():
    """K = 1, alpha = 0, unit strength: a plain LIF with constant drive c fires
    every p steps, p = min{k : c(1-b^k)/(1-b) >= theta}, and restarts at c."""
    b, theta = 0.5, 1.0
    for c in (0.55, 0.6, 0.7, 0.8, 1.2):
        p = next(k for k in range(1, 50) if c * (1 - b ** k) / (1 - b) >= theta)
        T = 4 * p + 1
        cfg = OracleConfig(T=T, K=1, G=1, C=1, psi="identity", reset="hard",
                           theta=theta, beta=b)
        s, v = run1(cfg, np.full((T, 1, 1), c))
        fired = np.nonzero(s[:, 0])[0] + 1
        assert list(fired) == list(range(p, T + 1, p)), (c, p, fired)
        for t0 in fired[:-1]:
            assert v[t0, 0] == pytest.approx(c, rel=1e-15)   # V^s[t0+1] = Z[t0+1]


def test_soft_reset_unrolled_sum():
    """Soft reset unrolled: V^s[t] = sum_{s<=t} b^{t-s} Z[s] - theta sum_{s<t} b^{t-s} S[s]."""
    rng = np.random.default_rng(5)
    T, b, theta = 12, 0.7, 1.0
    z = rng.uniform(0.0, 1.2, size=T)
    cfg = OracleConfig(T=T, K=1, G=1, C=1, psi="identity", reset="soft", theta=theta, beta=b)
    s, v = run1(cfg, z.reshape(T, 1, 1))
    s, v = s[:, 0], v[:, 0]
    assert s.any()
    for t in range(T):
        want = sum(b ** (t - u) * z[u] for u in range(t + 1)) - \
            theta * sum(b ** (t - u) * s[u] for u in range(t))
        assert v[t] == pytest.approx(want, rel=1e-12, abs=1e-14)
        assert s[t] == (1.0 if v[t] >= theta else 0.0)


# --------------------------------------------------------------------------- psi
def test_mexican_hat_is_minus_gaussian_second_derivative():
    xs = np.array([0.0, 0.1, 0.5, 1.0, 1.3, math.sqrt(3.0), 2.0, 2.7, 4.0])
    cfg = OracleConfig(T=1, K=1, G=1, C=1, psi="mh", reset="hard", theta=1e9, beta=0.0)
    _, v = run1(cfg, xs.reshape(1, -1, 1))
    g = lambda u: math.exp(-0.5 * u * u)
    h = 1e-4
    for x, got in zip(xs, v[0]):
        want = -(g(x + h) - 2 * g(x) + g(x - h)) / (h * h)
        assert got == pytest.approx(want, abs=2e-7), x
    assert v[0, 0] == 1.0                         # psi(0) = 1
    assert abs(v[0, 3]) < 1e-16                   # psi(1) = 0
    # even: negative input gives the same branch output
    _, vneg = run1(cfg, -xs.reshape(1, -1, 1))
    assert np.array_equal(v, vneg)


def test_mexican_hat_derivative_roots():
    """psi'(0) = psi'(sqrt 3) = 0: the gradient through a single MH branch vanishes there."""
    xs = np.array([[[0.0], [math.sqrt(3.0)], [1.0]]])
    cfg = OracleConfig(T=1, K=1, G=1, C=1, psi="mh", reset="hard", theta=1e9, beta=0.0)
    a, xi, z, k = one_neuron_params(1, 1)
    out = backward(cfg, xs, np.zeros(3, np.int32), None, a, xi, z, k, None,
                   np.zeros((1, 3)), np.ones((1, 3)))
    gx = out["gx"][0, :, 0]
    assert abs(gx[0]) < 1e-15 and abs(gx[1]) < 1e-15
    assert gx[2] == pytest.approx(-2.0 * math.exp(-0.5))    # psi'(1) = -2 e^{-1/2}


# --------------------------------------------------------------------------- L2 aggregation
def test_l2_branch_aggregation_pythagorean():
    cfg = OracleConfig(T=1, K=2, G=2, C=1, psi="identity", reset="hard", theta=1e9, beta=0.0)
    cases = [((3.0, 4.0), 0.0, 1.0, 5.0), ((5.0, 12.0), 0.0, 1.0, 13.0),
             ((4.0, 5.0), 1.0, 1.0, 5.0), ((3.0, 4.0), 0.0, 2.0, 2.5),
             ((-3.0, 4.0), 0.0, 1.0, 5.0)]
    for (x0, x1), xi, zeta, want in cases:
        _, v = run1(cfg, np.array([[[x0, x1]]]), xi=xi, zeta=zeta)
        assert v[0, 0] == want
    # G = 1 instead: two branches, Z = |3| + |4|
    cfg1 = OracleConfig(T=1, K=2, G=1, C=1, psi="identity", reset="hard", theta=1e9, beta=0.0)
    _, v = run1(cfg1, np.array([[[3.0, 4.0]]]))
    assert v[0, 0] == 7.0


# --------------------------------------------------------------------------- surrogate
def test_arctan_surrogate_values():
    """T = 1, Z = X: dL/dX = sg(X - theta) * gS with sg(0) = 1, sg(+-1/pi) = 1/2."""
    theta = 1.0
    xs = np.array([theta, theta + 1 / math.pi, theta - 1 / math.pi, theta + 2 / math.pi])
    cfg = OracleConfig(T=1, K=1, G=1, C=1, psi="identity", reset="hard", theta=theta, beta=0.5)
    a, xi, z, k = one_neuron_params(1, 1)
    out = backward(cfg, xs.reshape(1, -1, 1), np.zeros(4, np.int32), None, a, xi, z, k, None,
                   np.full((1, 4), 3.0))
    np.testing.assert_allclose(out["gx"][0, :, 0], [3.0, 1.5, 1.5, 3.0 / 5.0], rtol=1e-15)


def test_zero_norm_subgradient():
    """r_b = 0 (input exactly at xi): the branch passes zero gradient, no NaN."""
    cfg = OracleConfig(T=2, K=2, G=2, C=1, psi="identity", reset="hard", theta=1e9, beta=0.5)
    x = np.zeros((2, 1, 2))
    a, xi, z, k = one_neuron_params(2, 1, alpha=0.5)
    out = backward(cfg, x, np.zeros(1, np.int32), None, a, xi, z, k, None,
                   np.ones((2, 1)), np.ones((2, 1)))
    for key in ("gx", "galpha", "gxi", "gzeta"):
        assert np.all(out[key] == 0.0), key
    assert np.all(np.isfinite(out["gkappa"]))


# --------------------------------------------------------------------------- helpers
def random_case(rng, T, M, K, G, C, mask=False):
    Kb = K // G
    x = rng.normal(0.3, 1.0, size=(T, M, K))
    alpha = rng.uniform(0.5, 0.95, size=(C, K))
    xi = rng.normal(0.0, 0.1, size=(C, K))
    zeta = rng.uniform(0.8, 1.2, size=(C, Kb))
    kappa = rng.normal(1.0 / K, 0.1, size=(C, Kb)) + 0.4
    chan = rng.integers(0, C, size=M).astype(np.int32)
    m = None
    if mask:
        m = (rng.random((C, Kb)) < 0.5).astype(np.uint8)
        m[np.arange(C), rng.integers(0, Kb, size=C)] = 1     # keep one branch per channel
    return x, chan, alpha, xi, zeta, kappa, m


VARIANTS = [
    dict(K=1, G=1, psi="identity", reset="hard"),
    dict(K=2, G=1, psi="mh", reset="soft"),
    dict(K=2, G=2, psi="mh", reset="hard"),
    dict(K=4, G=1, psi="mh", reset="hard"),
    dict(K=4, G=2, psi="identity", reset="soft"),
    dict(K=4, G=4, psi="mh", reset="soft"),
    dict(K=4, G=2, psi="mh", reset="hard", stateless=True),
    dict(K=4, G=1, psi="identity", reset="hard", residual=True),
    dict(K=2, G=1, psi="mh", reset="hard", detach_reset=True),
]


def loss_and_grads_fd(cfg, x, chan, mrow, params, mask, ws, wv, h=1e-5):
    """Central differences of L = sum ws*S + sum wv*V w.r.t. x and each parameter."""
    def L(x_, p_):
        s, v = forward(cfg, x_, chan, mrow, *p_, mask)
        return float((ws * s).sum() + (wv * v).sum())

    gx = np.zeros_like(x)
    for idx in np.ndindex(*x.shape):
        xp, xm = x.copy(), x.copy()
        xp[idx] += h
        xm[idx] -= h
        gx[idx] = (L(xp, params) - L(xm, params)) / (2 * h)
    gp = []
    for j, p in enumerate(params):
        g = np.zeros_like(p)
        for idx in np.ndindex(*p.shape):
            pp = [q.copy() for q in params]
            pm = [q.copy() for q in params]
            pp[j][idx] += h
            pm[j][idx] -= h
            g[idx] = (L(x, pp) - L(x, pm)) / (2 * h)
        gp.append(g)
    return gx, gp


@pytest.mark.parametrize("var", VARIANTS, ids=lambda v: "-".join(f"{k}{v[k]}" for k in v))
@pytest.mark.parametrize("mode", ["subthreshold", "smooth_spike"])
def test_backward_matches_finite_differences(var, mode):
    if mode == "smooth_spike" and var.get("detach_reset"):
        pytest.skip("a detached reset is deliberately not the exact derivative")
    rng = np.random.default_rng(hash((mode, tuple(sorted(var.items())))) % 2**32)
    T, M, C = 5, 3, 2
    K, G = var["K"], var["G"]
    x, chan, alpha, xi, zeta, kappa, mask = random_case(rng, T, M, K, G, C, mask=True)
    if mode == "subthreshold":
        cfg = OracleConfig(T=T, K=K, G=G, C=C, theta=1e9, beta=0.6, **{
            k: v for k, v in var.items() if k not in ("K", "G")})
        ws = np.zeros((T, M))
    else:
        cfg = OracleConfig(T=T, K=K, G=G, C=C, theta=1.0, beta=0.6, smooth_spike=True, **{
            k: v for k, v in var.items() if k not in ("K", "G")})
        ws = rng.normal(size=(T, M))
    wv = rng.normal(size=(T, M))
    params = [alpha, xi, zeta, kappa]
    out = backward(cfg, x, chan, chan, *params, mask, ws, wv)
    fx, fp = loss_and_grads_fd(cfg, x, chan, chan, params, mask, ws, wv)
    np.testing.assert_allclose(out["gx"], fx, rtol=1e-6, atol=1e-8)
    for name, g in zip(("galpha", "gxi", "gzeta", "gkappa"), fp):
        if cfg.stateless and name == "galpha":
            assert np.all(out[name] == 0.0)
            continue
        np.testing.assert_allclose(out[name], g, rtol=1e-6, atol=1e-8, err_msg=name)
    # the somatic decay (learnable in a PLIF soma): beta is one number shared by every
    # channel, so finite differences see the sum of the per-channel gradients
    h = 1e-6

    def L_beta(b):
        s, v = forward(dataclasses.replace(cfg, beta=b), x, chan, chan, *params, mask)
        return float((ws * s).sum() + (wv * v).sum())

    fb = (L_beta(cfg.beta + h) - L_beta(cfg.beta - h)) / (2 * h)
    np.testing.assert_allclose(out["gbeta"].sum(), fb, rtol=1e-6, atol=1e-8)
    # and each channel's entry collects exactly its own neurons
    for c in range(C):
        own = (chan == c)[None, :]
        oc = backward(cfg, x, chan, chan, *params, mask, ws * own, wv * own)
        np.testing.assert_allclose(oc["gbeta"][c], out["gbeta"][c], rtol=1e-12, atol=1e-14)
        assert np.all(np.delete(oc["gbeta"], c) == 0.0)


def test_detach_reset_is_not_the_smooth_derivative():
    """With detach_reset the reset path is cut, so the gradient must differ from
    the full one (guards against the flag being ignored); its exact value is
    pinned by the autograd restatement, which detaches S in the reset term."""
    rng = np.random.default_rng(11)
    T, M, K, G, C = 5, 2, 2, 1, 1
    x, chan, alpha, xi, zeta, kappa, _ = random_case(rng, T, M, K, G, C)
    base = dict(T=T, K=K, G=G, C=C, psi="mh", reset="hard", theta=1.0, beta=0.6,
                smooth_spike=True)
    ws, wv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    full = backward(OracleConfig(**base), x, chan, None, alpha, xi, zeta, kappa, None, ws, wv)
    det = backward(OracleConfig(**base, detach_reset=True), x, chan, None, alpha, xi, zeta,
                   kappa, None, ws, wv)
    assert not np.allclose(full["gx"], det["gx"])


# --------------------------------------------------------------------------- autograd
class _Spike(torch.autograd.Function):
    """Heaviside forward, arctan-surrogate derivative backward (Eq. methods-sg)."""

    @staticmethod
    def forward(ctx, v_minus_theta):
        ctx.save_for_backward(v_minus_theta)
        return (v_minus_theta >= 0).to(v_minus_theta.dtype)

    @staticmethod
    def backward(ctx, g):
        (x,) = ctx.saved_tensors
        return g / (1 + (math.pi * x) ** 2)


def torch_dendsn(cfg, x, chan, mrow, alpha, xi, zeta, kappa, mask, beta=None):
    """Tensor restatement of the layer (float64 autograd), written independently
    of the C oracle: tensors over neurons, a Python loop over time. beta: the
    somatic decay as a tensor (to differentiate it), else cfg.beta."""
    beta = cfg.beta if beta is None else beta
    T, M, K = x.shape
    Kb, G = cfg.Kb, cfg.G
    a = torch.zeros_like(alpha[chan]) if cfg.stateless else alpha[chan]   # [M, K]
    ks = kappa[chan]                                                       # [M, Kb]
    if mask is not None:
        ks = ks * mask[torch.as_tensor(mrow, dtype=torch.long)].to(ks.dtype)
    vd = torch.zeros(M, K, dtype=x.dtype)
    vs = torch.zeros(M, dtype=x.dtype)
    sp = torch.zeros(M, dtype=x.dtype)
    S, V = [], []
    for t in range(T):
        vd = x[t] if cfg.stateless else a * vd + x[t]
        u = (vd - xi[chan]) / zeta[chan].repeat_interleave(G, dim=1)
        r = (u * u).reshape(M, Kb, G).sum(-1).sqrt()
        y = (1 - r * r) * torch.exp(-0.5 * r * r) if cfg.psi == "mh" else r
        z = (ks * y).sum(-1)
        if cfg.residual:
            z = z + x[t].mean(-1)
        sr = sp.detach() if cfg.detach_reset else sp
        if cfg.reset == "hard":
            vs = beta * (1 - sr) * vs + z
        else:
            vs = beta * (vs - cfg.theta * sr) + z
        sp = _Spike.apply(vs - cfg.theta)
        S.append(sp)
        V.append(vs)
    return torch.stack(S), torch.stack(V)


@pytest.mark.parametrize("var", VARIANTS + [
    dict(K=8, G=1, psi="mh", reset="soft"), dict(K=8, G=2, psi="identity", reset="hard")],
    ids=lambda v: "-".join(f"{k}{v[k]}" for k in v))
def test_backward_matches_autograd_restatement(var):
    rng = np.random.default_rng(sum(map(ord, str(sorted(var.items())))))
    T, M, C = 7, 40, 3
    K, G = var["K"], var["G"]
    x, chan, alpha, xi, zeta, kappa, mask = random_case(rng, T, M, K, G, C, mask=True)
    extra = {k: v for k, v in var.items() if k not in ("K", "G")}
    # threshold at the 70th percentile of the leak-only potential: plenty of spikes
    _, v_free = forward(OracleConfig(T=T, K=K, G=G, C=C, theta=1e9, beta=0.5, **extra),
                        x, chan, chan, alpha, xi, zeta, kappa, mask)
    theta = float(np.quantile(v_free, 0.7))
    cfg = OracleConfig(T=T, K=K, G=G, C=C, theta=theta, beta=0.5, **extra)
    gs = rng.normal(size=(T, M))
    gv = rng.normal(size=(T, M))
    s_o, v_o = forward(cfg, x, chan, chan, alpha, xi, zeta, kappa, mask)
    out = backward(cfg, x, chan, chan, alpha, xi, zeta, kappa, mask, gs, gv)

    tt = lambda a: torch.tensor(a, dtype=torch.float64, requires_grad=True)
    X, A, XI, Z, KA, BE = map(tt, (x, alpha, xi, zeta, kappa, cfg.beta))
    S, V = torch_dendsn(cfg, X, torch.as_tensor(chan, dtype=torch.long), chan, A, XI, Z, KA,
                        torch.as_tensor(mask), beta=BE)
    assert 0.05 < S.mean().item() < 0.95, "case should spike sometimes"
    # spike decisions can only differ where V sits on the threshold to rounding
    assert np.array_equal(S.detach().numpy(), s_o)
    np.testing.assert_allclose(V.detach().numpy(), v_o, rtol=1e-12, atol=1e-12)
    loss = (S * torch.as_tensor(gs)).sum() + (V * torch.as_tensor(gv)).sum()
    loss.backward()
    np.testing.assert_allclose(out["gx"], X.grad.numpy(), rtol=1e-10, atol=1e-12)
    ga = np.zeros_like(alpha) if cfg.stateless else A.grad.numpy()
    np.testing.assert_allclose(out["galpha"], ga, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(out["gxi"], XI.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(out["gzeta"], Z.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(out["gkappa"], KA.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(out["gbeta"].sum(), BE.grad.item(), rtol=1e-10, atol=1e-12)


# --------------------------------------------------------------------------- invariants
def test_kappa_linearity_and_mask_equals_zero_strength():
    rng = np.random.default_rng(3)
    T, M, K, G, C = 6, 10, 4, 1, 2
    x, chan, alpha, xi, zeta, kappa, _ = random_case(rng, T, M, K, G, C)
    cfg = OracleConfig(T=T, K=K, G=G, C=C, psi="mh", reset="hard", theta=1e9, beta=0.0)
    _, v1 = forward(cfg, x, chan, None, alpha, xi, zeta, kappa)
    _, v2 = forward(cfg, x, chan, None, alpha, xi, zeta, 2.0 * kappa)
    assert np.array_equal(2.0 * v1, v2)                 # beta = 0: V = Z, linear in kappa

    cfg = OracleConfig(T=T, K=K, G=G, C=C, psi="mh", reset="hard", theta=1.0, beta=0.5)
    mask = np.ones((C, K), np.uint8)
    mask[0, 1] = 0
    mask[1, 3] = 0
    k0 = kappa.copy()
    k0[0, 1] = 0.0
    k0[1, 3] = 0.0
    gs, gv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    sm, vm = forward(cfg, x, chan, chan, alpha, xi, zeta, kappa, mask)
    sz, vz = forward(cfg, x, chan, None, alpha, xi, zeta, k0)
    assert np.array_equal(sm, sz) and np.array_equal(vm, vz)
    bm = backward(cfg, x, chan, chan, alpha, xi, zeta, kappa, mask, gs, gv)
    for c, b in ((0, 1), (1, 3)):
        sel = chan == c
        assert np.all(bm["gx"][:, sel, b] == 0.0)
        assert bm["galpha"][c, b] == 0 and bm["gxi"][c, b] == 0
        assert bm["gzeta"][c, b] == 0 and bm["gkappa"][c, b] == 0
    assert np.any(bm["gkappa"] != 0)


def test_identical_branches_equal_one_scaled_branch():
    rng = np.random.default_rng(4)
    T, M = 8, 6
    x1 = rng.normal(0.3, 1.0, size=(T, M, 1))
    cfg1 = OracleConfig(T=T, K=1, G=1, C=1, psi="mh", reset="hard", theta=1.0, beta=0.5)
    cfg4 = OracleConfig(T=T, K=4, G=1, C=1, psi="mh", reset="hard", theta=1.0, beta=0.5)
    z = np.zeros(M, np.int32)
    s1, v1 = forward(cfg1, x1, z, None, [[0.7]], [[0.05]], [[0.9]], [[4 * 0.3]])
    s4, v4 = forward(cfg4, np.repeat(x1, 4, axis=2), z, None, [[0.7] * 4], [[0.05] * 4],
                     [[0.9] * 4], [[0.3] * 4])
    np.testing.assert_allclose(v4, v1, rtol=1e-14, atol=1e-15)
    assert np.array_equal(s1, s4)


def test_stateless_equals_stateful_with_zero_decay():
    rng = np.random.default_rng(6)
    T, M, K, G, C = 6, 8, 4, 2, 2
    x, chan, alpha, xi, zeta, kappa, _ = random_case(rng, T, M, K, G, C)
    gs, gv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    c_sl = OracleConfig(T=T, K=K, G=G, C=C, psi="mh", reset="soft", stateless=True)
    c_sf = OracleConfig(T=T, K=K, G=G, C=C, psi="mh", reset="soft")
    a = forward(c_sl, x, chan, None, alpha, xi, zeta, kappa)
    b = forward(c_sf, x, chan, None, np.zeros_like(alpha), xi, zeta, kappa)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    ga = backward(c_sl, x, chan, None, alpha, xi, zeta, kappa, None, gs, gv)
    gb = backward(c_sf, x, chan, None, np.zeros_like(alpha), xi, zeta, kappa, None, gs, gv)
    for k in ("gx", "gxi", "gzeta", "gkappa"):
        np.testing.assert_array_equal(ga[k], gb[k])
    assert np.all(ga["galpha"] == 0)


def test_residual_with_zero_strength_is_lif_on_mean_input():
    T = 7
    cfg = OracleConfig(T=T, K=2, G=1, C=1, psi="mh", reset="hard", theta=1.0, beta=0.5,
                       residual=True)
    x = np.tile(np.array([0.25, 1.0]), (T, 1, 1))     # mean 0.625: the golden plain-LIF case
    s, v = run1(cfg, x, kappa=0.0)
    np.testing.assert_array_equal(v[:, 0], [0.625, 0.9375, 1.09375] * 2 + [0.625])
    np.testing.assert_array_equal(s[:, 0], [0, 0, 1, 0, 0, 1, 0])


def test_parameter_gradients_sum_over_channel_members():
    rng = np.random.default_rng(8)
    T, M, K, G, C = 5, 9, 4, 2, 3
    x, chan, alpha, xi, zeta, kappa, mask = random_case(rng, T, M, K, G, C, mask=True)
    cfg = OracleConfig(T=T, K=K, G=G, C=C, psi="mh", reset="hard")
    gs, gv = rng.normal(size=(T, M)), rng.normal(size=(T, M))
    full = backward(cfg, x, chan, chan, alpha, xi, zeta, kappa, mask, gs, gv)
    acc = {k: np.zeros_like(full[k]) for k in ("galpha", "gxi", "gzeta", "gkappa")}
    for m in range(M):
        one = backward(cfg, x[:, m:m + 1], chan[m:m + 1], chan[m:m + 1], alpha, xi, zeta,
                       kappa, mask, gs[:, m:m + 1], gv[:, m:m + 1])
        np.testing.assert_array_equal(one["gx"][:, 0], full["gx"][:, m])
        for k in acc:
            acc[k] += one[k]
        c = chan[m]
        for k in acc:                       # other channels untouched
            other = np.delete(one[k], c, axis=0)
            assert np.all(other == 0)
    for k in acc:
        np.testing.assert_allclose(full[k], acc[k], rtol=1e-12, atol=1e-14)


def test_layer_channel_map():
    chan, mrow = layer_channels(B=2, N=8, C=2, inner=4, mask_per_neuron=False)
    assert chan.tolist() == [0, 0, 0, 0, 1, 1, 1, 1] * 2
    assert mrow.tolist() == chan.tolist()
    chan, mrow = layer_channels(B=2, N=8, C=4, inner=1, mask_per_neuron=True)
    assert chan.tolist() == [0, 1, 2, 3, 0, 1, 2, 3] * 2
    assert mrow.tolist() == list(range(8)) * 2


def test_paper_layout_reader_places_each_compartment():
    """(C_o, P, H, W) grouping: compartment k of neuron n = g*inner + s sits at [g, k, s]."""
    from types import SimpleNamespace
    from oracle import layer_x
    T, B, N, K, inner = 2, 2, 6, 2, 3
    w = SimpleNamespace(T=T, B=B, N=N, K=K, inner=inner, layout="paper")
    xp = np.zeros((T, B, N // inner, K, inner))
    for t in range(T):
        for b in range(B):
            for g in range(N // inner):
                for k in range(K):
                    for s in range(inner):
                        xp[t, b, g, k, s] = 1000 * t + 100 * b + 10 * (g * inner + s) + k
    got = layer_x(w, xp).reshape(T, B, N, K)
    t, b, n, k = np.meshgrid(*[np.arange(d) for d in (T, B, N, K)], indexing="ij")
    assert np.array_equal(got, 1000 * t + 100 * b + 10 * n + k)


def test_paper_layout_gives_the_same_layer():
    """The same draws in either layout give the same spikes and (permuted) gradients."""
    from oracle import backward_layer, forward_layer
    from paper_2412_06355_gb300 import workloads
    w = workloads.Workload("lay", T=5, B=2, N=2 * 3 * 4, K=4, G=2, C=3, inner=4, dtype="f32",
                           psi="mh", reset="hard", seed=11)
    wp = w.with_(layout="paper")
    a, ap = workloads.make_inputs(w, with_gv=True), workloads.make_inputs(wp, with_gv=True)
    assert tuple(ap["x"].shape) == (5, 2, 2 * 3, 4, 4)
    s, v = forward_layer(w, a)
    sp, vp = forward_layer(wp, ap)
    assert np.array_equal(s, sp) and np.array_equal(v, vp)
    g, gp = backward_layer(w, a), backward_layer(wp, ap)
    gx_back = gp["gx"].transpose(0, 1, 2, 4, 3).reshape(g["gx"].shape)
    assert np.array_equal(g["gx"], gx_back)
    for k in ("galpha", "gxi", "gzeta", "gkappa"):
        assert np.array_equal(g[k], gp[k])
