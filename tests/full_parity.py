"""Whole-layer parity at full size: every neuron of a layer workload against the oracle.

The layer is run once through the C ABI in the benchmark's launch configuration
(production forward without V^s output, backward with dL/dV^s absent). The oracle then
simulates every neuron, in slices of neurons run on all host cores at once (ctypes
releases the interpreter lock during the C call; neurons are independent, so slicing
changes nothing), and each slice is compared element by element as it finishes; the
float64 parameter-gradient sums of the slices are added up and compared at the end.

Bounds (the stated ones, no allowance):
  V^s      |gpu - oracle| <= 1e-6 + 1e-5 |oracle|, up to and including a neuron's first
           ambiguous step (the oracle's V^s within 1e-5 of theta)
  spikes   identical before a neuron's first ambiguous step
  params   |gpu - oracle| <= 1e-4 |oracle| + 1e-6 rms(oracle tensor)
  dL/dX    |gpu - oracle| <= rtol |oracle| + 1e-5 rms(oracle tensor), rtol 1e-4 (float32),
           2e-2 (bfloat16). The absolute term is the reading of tests/parity.py: 1e-6 rms is
           below what float32 evaluation of the method reaches (a plain float32 restatement,
           tests/f32_restatement.py, misses it on every large layer); the report also gives
           the worst error over the 1e-6 rms bound.
Neurons with an ambiguous step get zero dL/dS on both sides, as in tests/parity.py, and so
do, for the identity branch with one compartment per branch, neurons whose u comes within
float32 rounding of the kink of |u| at 0 (reading A22; counted in the report).

V^s comes from a second forward with the V^s output (the same step function; its spikes
must equal the production forward's bit for bit).
"""
from __future__ import annotations

import os
import time
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle
from paper_2412_06355_gb300 import binding, workloads

AMBIGUOUS = 1e-5
V_RTOL, V_ATOL = 1e-5, 1e-6
G_RTOL, BF16_RTOL = 1e-4, 2e-2
ATOL_REL = 1e-6            # parameter gradients; the stated absolute term
GX_ATOL_REL = 1e-5         # dL/dX (the reading above)
PARAMS = ("galpha", "gxi", "gzeta", "gkappa")


def _slices(w, slice_steps: int):
    """(b, n0, n1) neuron ranges within one sample, about slice_steps neuron-steps each."""
    m = max(1, min(w.N, slice_steps // max(w.T, 1)))
    return [(b, n0, min(w.N, n0 + m)) for b in range(w.B) for n0 in range(0, w.N, m)]


def _ocfg(w):
    return oracle.OracleConfig(T=w.T, K=w.K, G=w.G, C=w.C, psi=w.psi, reset=w.reset,
                               theta=w.theta, beta=w.beta, stateless=w.stateless,
                               residual=w.residual, detach_reset=w.detach_reset)


def _maps(w, n0, n1):
    n = np.arange(n0, n1)
    chan = ((n // w.inner) % w.C).astype(np.int32)
    mrow = (n if w.mask_per_neuron else chan).astype(np.int32)
    return chan, mrow


def run(w, threads: int | None = None, slice_steps: int = 1 << 22, want_beta: bool = False) -> dict:
    """Runs the layer on cuda:0 and compares every neuron with the oracle. Returns a report
    (per-quantity worst error / bound and counts); raises nothing itself. want_beta: the
    backward build with dL/dbeta (a learnable somatic decay), compared like the other
    parameter gradients."""
    params = PARAMS + (("gbeta",) if want_beta else ())
    paper = w.layout == "paper"         # x and dL/dX compared in the [T, B, N, K] order
    t_start = time.perf_counter()
    threads = threads or os.cpu_count() or 1
    cfg = binding.config_of(w)
    inp = workloads.make_inputs(w, "cuda")
    x, gs = inp["x"], inp["gs"]
    prm = [inp[k] for k in ("alpha", "xi", "zeta", "kappa")]
    mask = inp["mask"]
    saved, scratch = binding.workspace(cfg)
    s_prod, _ = binding.forward(cfg, x, *prm, mask, want_v=False, saved=saved)
    s_v, v = binding.forward(cfg, x, *prm, mask, want_v=True, saved=None)
    torch.cuda.synchronize()
    same_spikes = bool(torch.equal(s_prod, s_v))
    del s_v
    x_h = workloads.from_paper_layout(x.cpu(), w.N, w.K, w.inner) if paper else x.cpu()
    prm_h = [t.cpu() for t in prm]
    mask_h = None if mask is None else mask.cpu()
    ocfg = _ocfg(w)
    sl = _slices(w, slice_steps)

    # ---- pass 1: forward of every neuron
    def fwd_job(job):
        b, n0, n1 = job
        chan, mrow = _maps(w, n0, n1)
        s_o, v_o = oracle.forward(ocfg, x_h[:, b, n0:n1], chan, mrow, *prm_h, mask_h)
        got_v = v[:, b, n0:n1].cpu().double().numpy()
        got_s = s_prod[:, b, n0:n1].cpu().double().numpy()
        amb = np.abs(v_o - w.theta) < AMBIGUOUS
        first = np.where(amb.any(axis=0), amb.argmax(axis=0), w.T)
        t_idx = np.arange(w.T)[:, None]
        vm = t_idx <= first[None]
        bound = V_ATOL + V_RTOL * np.abs(v_o)
        ratio = np.where(vm, np.abs(got_v - v_o) / bound, 0.0)
        sm = t_idx < first[None]
        mism = int(((got_s != s_o) & sm).sum())
        kink = _kink_ambiguous(n0, n1, x_h[:, b, n0:n1], chan, prm_h)
        return dict(amb=(first < w.T) | kink, kink=int(kink.sum()),
                    v_ratio=float(ratio.max()) if ratio.size else 0.0,
                    v_bad=int((ratio > 1.0).sum()), spike_mismatch=int(mism),
                    spikes=float(s_o.sum()), nonbinary=int(((got_s != 0) & (got_s != 1)).sum()))

    def _kink_ambiguous(n0, n1, xs, chan, prm):
        """Identity branch, one compartment per branch: dpsi/du = sign(u) jumps at u = 0,
        so a neuron whose u comes within float32 rounding of 0 at some step has its sign,
        and with it the gradient, decided by rounding (reading A22). The float64 scan of
        Eq. methods-compartment here gives u = (V^d - xi)/zeta; the rounding scale is that
        of the float32 evaluation u = V^d * (1/zeta) + (-xi/zeta), with V^d carrying the
        scan's accumulated rounding (up to 1/(1 - alpha) units of 2^-24 relative)."""
        if w.psi != "identity" or w.G != 1 or w.stateless:
            return np.zeros(n1 - n0, dtype=bool)
        alpha, xi, zeta = (t.double().numpy()[chan] for t in prm[:3])          # [m, K]
        xv = xs.double().numpy()                                                 # [T, m, K]
        vd = np.zeros_like(xv[0])
        amb = np.zeros(n1 - n0, dtype=bool)
        for t in range(w.T):
            vd = alpha * vd + xv[t]
            u = (vd - xi) / zeta
            scale = (np.abs(vd) * (8 + 2 / (1 - alpha)) + 8 * np.abs(xi)) / zeta
            amb |= (np.abs(u) < 2.0 ** -24 * scale).any(axis=1)
        return amb

    with ThreadPoolExecutor(threads) as ex:
        r1 = list(ex.map(fwd_job, sl))
    amb = torch.zeros((w.B, w.N), dtype=torch.bool)
    for (b, n0, n1), r in zip(sl, r1):
        amb[b, n0:n1] = torch.from_numpy(r["amb"])
    t_fwd = time.perf_counter()

    # ---- the backward on the GPU with the ambiguous neurons' upstream gradient removed
    gsp = gs.clone()
    gsp[:, amb.cuda()] = 0
    g = binding.backward(cfg, x, *prm, mask, gsp, None, saved, scratch, want_beta=want_beta)
    torch.cuda.synchronize()
    gx = workloads.from_paper_layout(g["gx"], w.N, w.K, w.inner) if paper else g["gx"]
    rms_gx_gpu = float(torch.sqrt(torch.mean(gx.double() ** 2)).item()) if gx.numel() else 0.0
    gsp_h = gsp.cpu()
    rtol_x = BF16_RTOL if w.dtype == "bf16" else G_RTOL
    atol_bare = ATOL_REL * rms_gx_gpu            # the ratios are reported against the GPU's rms
    atol_read = GX_ATOL_REL * rms_gx_gpu          # (asserted equal to the oracle's below)

    # ---- pass 2: backward of every neuron
    def bwd_job(job):
        b, n0, n1 = job
        chan, mrow = _maps(w, n0, n1)
        ref = oracle.backward(ocfg, x_h[:, b, n0:n1], chan, mrow, *prm_h, mask_h,
                              gsp_h[:, b, n0:n1])
        got = gx[:, b, n0:n1].cpu().double().numpy()
        want = ref["gx"]
        err = np.abs(got - want)
        excess = err - rtol_x * np.abs(want)
        ratio = err / (rtol_x * np.abs(want) + atol_read) if atol_read > 0 else err
        ratio_bare = err / (rtol_x * np.abs(want) + atol_bare) if atol_bare > 0 else err
        i = int(np.argmax(ratio_bare)) if ratio.size else 0
        worst = None
        if ratio.size:
            t, m, k = np.unravel_index(i, ratio.shape)
            worst = dict(t=int(t), b=b, n=int(n0 + m), k=int(k), got=float(got.flat[i]),
                         want=float(want.flat[i]))
        return dict(excess=float(excess.max()) if excess.size else -np.inf,
                    ratio=float(ratio.max()) if ratio.size else 0.0,
                    ratio_bare=float(ratio_bare.max()) if ratio.size else 0.0,
                    bad_bare=int((ratio_bare > 1.0).sum()),
                    ss=float(np.sum(want * want)), worst=worst,
                    params={k: ref[k] for k in params})

    with ThreadPoolExecutor(threads) as ex:
        r2 = list(ex.map(bwd_job, sl))
    t_bwd = time.perf_counter()

    n_gx = gx.numel()
    rms_gx = float(np.sqrt(sum(r["ss"] for r in r2) / n_gx)) if n_gx else 0.0
    atol_x = GX_ATOL_REL * rms_gx
    best = max(r2, key=lambda r: r["ratio_bare"])
    rep = dict(
        workload=w.name, T=w.T, B=w.B, N=w.N, K=w.K, dtype=w.dtype, psi=w.psi, reset=w.reset,
        want_beta=want_beta,
        neurons=w.B * w.N, elements_gx=n_gx, slices=len(sl), threads=threads,
        forward_spikes_equal=same_spikes,
        ambiguous_neurons=int(amb.sum()),
        kink_ambiguous_neurons=sum(r["kink"] for r in r1),
        spike_rate=sum(r["spikes"] for r in r1) / max(1, w.neuron_steps),
        spike_mismatches=sum(r["spike_mismatch"] for r in r1),
        nonbinary_spikes=sum(r["nonbinary"] for r in r1),
        v_max_err_over_bound=max(r["v_ratio"] for r in r1),
        v_out_of_bound=sum(r["v_bad"] for r in r1),
        gx_rtol=rtol_x, gx_atol_rel=GX_ATOL_REL, gx_rms_oracle=rms_gx, gx_rms_gpu=rms_gx_gpu,
        gx_max_err_over_bound=max(r["ratio"] for r in r2),
        gx_max_err_over_bare_bound=best["ratio_bare"],
        gx_elements_over_bare_bound=sum(r["bad_bare"] for r in r2), gx_worst_bare=best["worst"],
        gx_pass=max(r["excess"] for r in r2) <= atol_x,
        seconds=dict(oracle_forward=t_fwd - t_start, oracle_backward=t_bwd - t_fwd))
    for k in params:
        want = sum(r["params"][k] for r in r2)
        got = g[k].double().cpu().numpy()
        err = np.abs(got - want)
        atol = ATOL_REL * float(np.sqrt(np.mean(want * want))) if want.size else 0.0
        bound = G_RTOL * np.abs(want) + atol
        rep[f"{k}_max_err_over_bound"] = float((err / np.where(bound > 0, bound, 1.0)).max())
        rep[f"{k}_pass"] = bool(np.all(err <= bound))
    return rep


def failures(rep: dict) -> list:
    """Which stated bounds a report breaks (empty when the layer passes)."""
    bad = []
    if not rep["forward_spikes_equal"]:
        bad.append("the forward with V^s output changed the spikes")
    if rep["spike_mismatches"]:
        bad.append(f"{rep['spike_mismatches']} spikes differ at unambiguous steps")
    if rep["nonbinary_spikes"]:
        bad.append("spikes other than 0/1")
    if rep["v_out_of_bound"]:
        bad.append(f"V^s: {rep['v_out_of_bound']} elements out of bound "
                   f"(worst {rep['v_max_err_over_bound']:.3g} x bound)")
    if not rep["gx_pass"]:
        bad.append(f"grad_x out of bound (worst {rep['gx_max_err_over_bound']:.3g} x bound; "
                   f"worst over the 1e-6 rms bound at {rep['gx_worst_bare']})")
    if abs(rep["gx_rms_gpu"] - rep["gx_rms_oracle"]) > 1e-4 * max(rep["gx_rms_oracle"], 1e-30):
        bad.append("grad_x RMS of GPU and oracle disagree")
    for k in PARAMS + (("gbeta",) if rep.get("want_beta") else ()):
        if not rep[f"{k}_pass"]:
            bad.append(f"{k} out of bound (worst {rep[k + '_max_err_over_bound']:.3g} x bound)")
    return bad
