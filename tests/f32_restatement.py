"""A plain float32 restatement of the DendSN layer's forward and backward (test tool).

It computes what the oracle computes, in the same order (Eqs. methods-compartment ..
methods-lif-fire forward, the chain rule of the oracle's backward in reverse time), but
with every intermediate rounded to float32: each product, sum and quotient is one IEEE
float32 operation (no fused multiply-add), and e^x is the float64 exponential rounded to
float32 (correctly rounded up to double rounding). It is vectorised over neurons and
shares no code with the oracle or the CUDA library.

Its only use is to measure what float32 arithmetic itself does to the results: where
even this restatement misses a bound against the float64 oracle, that bound is tighter
than float32 evaluation of the method allows, whatever the implementation. Supports
G = 1 and G > 1, both branch nonlinearities, both resets, per-neuron or per-channel
masks, the Stateless and residual dendrites.
"""
from __future__ import annotations

import numpy as np

F = np.float32
PI = F(np.pi)


def _exp(z: np.ndarray) -> np.ndarray:
    return np.exp(z.astype(np.float64)).astype(F)


def _params(w, inp, chan, mrow):
    f = lambda k: np.asarray(inp[k].float().cpu().numpy() if hasattr(inp[k], "cpu") else inp[k], F)
    a, xi = f("alpha")[chan], f("xi")[chan]                 # [M, K]
    ze, ka = f("zeta")[chan], f("kappa")[chan]              # [M, Kb]
    m = np.ones_like(ka)
    if inp.get("mask") is not None:
        mk = inp["mask"].cpu().numpy() if hasattr(inp["mask"], "cpu") else inp["mask"]
        m = np.asarray(mk, F)[mrow]
    return a, xi, ze, ka, m


def run(w, x, inp, chan, mrow, gs, gv=None):
    """x [T, M, K], gs (and gv) [T, M]: any float dtype (converted exactly to float32).
    Returns dict v, s [T, M], gx [T, M, K] as float32, and per-neuron-summed parameter
    gradients galpha, gxi [C, K], gzeta, gkappa [C, Kb] (float64 sums of float32 terms)."""
    T, M, K = x.shape
    G, Kb = w.G, w.K // w.G
    x = np.asarray(x, F)
    gs = np.asarray(gs, F)
    gv = None if gv is None else np.asarray(gv, F)
    a, xi, ze, ka, m = _params(w, inp, chan, mrow)
    if w.stateless:
        a = np.zeros_like(a)                                 # V^d = X
    km = ka * m
    zr = np.repeat(ze, G, axis=1)
    beta, theta = F(w.beta), F(w.theta)
    mh = w.psi == "mh"
    vd_h = np.zeros((T + 1, M, K), F)
    u_h = np.zeros((T, M, K), F)
    r_h = np.zeros((T, M, Kb), F)
    y_h = np.zeros((T, M, Kb), F)
    v_h = np.zeros((T, M), F)
    s_h = np.zeros((T, M), bool)
    v = np.zeros(M, F)
    s = np.zeros(M, bool)
    for t in range(T):
        vd = a * vd_h[t] + x[t]
        vd_h[t + 1] = vd
        u = (vd - xi) / zr
        u_h[t] = u
        if G == 1:
            r = np.abs(u)
        else:
            sq = u[:, 0::G] * u[:, 0::G]
            for q in range(1, G):
                sq = sq + u[:, q::G] * u[:, q::G]
            r = np.sqrt(sq)
        y = (F(1) - r * r) * _exp(-(r * r) / F(2)) if mh else r
        r_h[t], y_h[t] = r, y
        z = km[:, 0] * y[:, 0]
        for b in range(1, Kb):
            z = z + km[:, b] * y[:, b]
        if w.residual:                                      # Eq. methods-residual
            xs = x[t][:, 0]
            for i in range(1, K):
                xs = xs + x[t][:, i]
            z = z + xs / F(K)
        if w.reset == "hard":
            v = np.where(s, F(0), beta * v) + z
        else:
            v = beta * (v - np.where(s, theta, F(0))) + z
        s = v >= theta
        v_h[t], s_h[t] = v, s

    gx = np.zeros((T, M, K), F)
    A = np.zeros((M, K), F)
    dvn = np.zeros(M, F)
    ga = np.zeros((M, K), F)
    gxi = np.zeros((M, K), F)
    gz = np.zeros((M, Kb), F)
    gk = np.zeros((M, Kb), F)
    for t in range(T - 1, -1, -1):
        if w.detach_reset:
            dnds = np.zeros(M, F)
        elif w.reset == "hard":
            dnds = -(beta * v_h[t])
        else:
            dnds = np.full(M, -(beta * theta), F)
        dndv = np.where(s_h[t], F(0), beta) if w.reset == "hard" else np.full(M, beta, F)
        dS = gs[t] + dnds * dvn
        xs = v_h[t] - theta
        sg = F(1) / (F(1) + (PI * PI) * (xs * xs))
        dV = sg * dS + dndv * dvn
        if gv is not None:
            dV = dV + gv[t]
        dY = km * dV[:, None]
        r = r_h[t]
        if mh:
            dr = r * (r * r - F(3)) * _exp(-(r * r) / F(2)) * dY
        else:
            dr = dY
        u = u_h[t]
        rr = np.repeat(r, G, axis=1)
        dr_rep = np.repeat(dr, G, axis=1)
        safe = np.where(rr > 0, rr, F(1))
        du = np.where(rr > 0, dr_rep * u / safe, F(0))
        direct = du / zr
        A = direct + a * A
        gx[t] = A + dV[:, None] / F(K) if w.residual else A
        ga = ga + A * vd_h[t]
        gxi = gxi - direct
        gz = gz - dr * r / ze
        gk = gk + m * y_h[t] * dV[:, None]
        dvn = dV
    C = w.C
    out = dict(v=v_h, s=s_h.astype(F), gx=gx)
    for k, arr, width in (("galpha", ga, K), ("gxi", gxi, K), ("gzeta", gz, Kb),
                          ("gkappa", gk, Kb)):
        acc = np.zeros((C, width))
        np.add.at(acc, chan, arr.astype(np.float64))
        out[k] = acc
    return out
