#!/usr/bin/env python
"""Throughput of the fused DendSN layer step (forward + BPTT backward) on GB300.

One step = dendsn_forward + dendsn_backward over one batch of the workload (all of
x read, spikes written, grad_x and the four parameter gradients produced); with N
ranks (torchrun) every rank processes its own batch and the parameter gradients
are summed with one all-reduce (weak scaling).

The headline is the long-horizon event-stream layer (T=64, B=32, 128 x 32 x 32
neurons, K=4, float32, 80% zero inputs), the largest of the layer workloads. The
same JSON line carries one block per other large layer workload (the conv layer,
the deeper bf16 conv layer and the transformer-token layer with branch gating),
each timed, roofline-checked and CPU-baselined the same way.

Prints ONE JSON line on rank 0. Everything else goes to stderr.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload event]
                  [--blocks conv,deepconv_bf16,token_dbg] [--impl ours|reference]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "DendSN fwd+bwd neuron-timesteps/sec and achieved HBM GB/s vs 8 TB/s (1 GB300)"
UNIT = "neuron-steps/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 2**20
FP32_LANES_PER_SM = 128          # float32 FMA lanes per Blackwell SM
NOMINAL_SM_MHZ = 2070.0
HEADLINE = "event"
BLOCKS = ("conv", "deepconv_bf16", "token_dbg")


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--graph", action="store_true",
                    help="replay the forward and backward as captured CUDA graphs")
    ap.add_argument("--plif", action="store_true",
                    help="learnable somatic decay: time dendsn_backward_plif (adds dL/dbeta)")
    ap.add_argument("--no-lif", action="store_true",
                    help="skip timing the point-neuron LIF layer baseline")
    ap.add_argument("--workload", default=HEADLINE)
    ap.add_argument("--blocks", default=None,
                    help="comma-separated layer workloads timed after the headline and reported "
                         "as blocks of the same line (default: the other large layers when the "
                         "headline is the default one, else none; 'none' for none)")
    ap.add_argument("--psi", choices=["mh", "identity"], default=None)
    ap.add_argument("--batch", type=int, default=None,
                    help="override the workload's batch B (smaller profiling captures)")
    ap.add_argument("--variant", choices=["stateful", "stateless", "resstateless", "resstateful"],
                    default="stateful", help="dendrite variant (Methods, DendSN variants)")
    ap.add_argument("--cpu-seconds", type=float, default=8.0,
                    help="target CPU time of the oracle baseline sample of each layer")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def measured_hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clock/throttle samples with GPU timestamps, filtered to a window."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except FileNotFoundError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.out.flush()
        self.out.seek(0)
        rows = []
        for line in self.out.read().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S")) + \
                    float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append(dict(t=ts, sm=float(parts[2]), sm_max=float(parts[3]),
                                 power=float(parts[4]) if parts[4] not in ("[N/A]", "N/A") else None,
                                 reasons={"hw_slowdown": parts[6], "hw_thermal_slowdown": parts[7],
                                          "sw_thermal_slowdown": parts[8],
                                          "sw_power_cap": parts[9]}))
            except (ValueError, IndexError):
                continue
        os.unlink(self.out.name)
        return rows

    @staticmethod
    def summarize(rows, t0, t1):
        win = [r for r in rows if t0 - 0.1 <= r["t"] <= t1 + 0.1]
        note = "samples inside the timed region"
        if not win:
            load = [r for r in rows if r["sm"] > 0.5 * r["sm_max"]]
            win = load or rows
            note = "timed region shorter than the sampling period: samples from the loaded run"
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi unavailable"}
        reasons = sorted({k for r in win for k, v in r["reasons"].items() if v == "Active"})
        return {"sm_mhz": statistics.median(r["sm"] for r in win),
                "sm_max_mhz": max(r["sm_max"] for r in win), "reasons": reasons,
                "samples": len(win), "note": note}


# ------------------------------------------------------------------ kernel names
def kernel_names(w):
    """(forward, backward) kernels the library launches for workload w, following its plan:
    narrow long-horizon layers take the time-parallel kernels; rows of one full chunk
    (T = 4 or 8) whose 8 compartments sit on one lane, compartments innermost and no
    residual term, take the phased backward (one lane per neuron: bf16, or float32 with
    8-step chunks; for bf16 the build that reads the V^s its forward kept in the saved
    buffer, which the benchmark always provides); 4-step rows of 8 float32 compartments on
    two lanes (no residual term, either layout) the row-pair backward; the rest the chunked
    kernels."""
    if w.T >= 256 and w.B * w.N <= 2048:
        return "tp_forward_kernel", "tp_backward_kernel"
    L = 4 if w.T <= 4 else 8
    layout0 = w.layout == "kinner" or w.K == 1 or w.inner == 1
    staged = (not layout0 and 2 <= w.K <= 8 and w.inner % 32 == 0)
    fwd = "dendsn_forward_staged_kernel" if staged else "dendsn_forward_kernel"
    one_lane = w.K == 8 and w.G == 1 and (w.dtype == "bf16" or L == 8)
    if one_lane and layout0 and w.T == L and not w.residual:
        return fwd, ("dendsn_backward_phased_vs_kernel" if w.dtype == "bf16"
                     else "dendsn_backward_phased_kernel")
    if w.K == 8 and w.G == 1 and w.dtype == "f32" and w.T == 4 and not w.residual:
        return fwd, "dendsn_backward_rowpair_kernel"
    return fwd, "dendsn_backward_kernel"


# ------------------------------------------------------------------ traffic record
def _strip_comments(src: str) -> str:
    """C/C++ source without // and /* */ comments and blank lines (comments do not change
    the compiled kernels, so they must not invalidate recorded counters)."""
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    return "\n".join(line.rstrip() for line in src.splitlines() if line.strip())


def kernel_source_hash():
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2412_06355_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh", ".h")):
            with open(os.path.join(csrc, name), encoding="utf-8") as f:
                h.update(name.encode() + _strip_comments(f.read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if the kernel is unchanged."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    ent = rec.get(workload, {}).get(kernel)
    if not ent or ent.get("source_hash") != kernel_source_hash():
        return None
    return ent.get("dram_bytes_per_launch")


# ------------------------------------------------------------------ oracle (CPU baseline)
def host_cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the platform string)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            k, _, v = line.partition(":")
            if k.strip() == "Model name" and v.strip():
                vendor = next((l.partition(":")[2].strip() for l in out.splitlines()
                               if l.partition(":")[0].strip() == "Vendor ID"), "")
                return f"{vendor} {v.strip()}".strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                k, _, v = line.partition(":")
                if k.strip().lower() in ("model name", "cpu model") and v.strip():
                    return v.strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


class pinned_to_one_core:
    """Runs the enclosed block with this process restricted to one host core (the last one
    it may use), then restores its affinity. Yields the core (None where affinity is not
    available)."""

    def __enter__(self):
        self.saved = None
        self.core = None
        if hasattr(os, "sched_getaffinity"):
            self.saved = os.sched_getaffinity(0)
            self.core = max(self.saved)
            os.sched_setaffinity(0, {self.core})
        return self.core

    def __exit__(self, *exc):
        if self.saved is not None:
            os.sched_setaffinity(0, self.saved)
        return False


def oracle_sample_rate(w, inp_cpu_fn, target_s: float):
    """Times the float64 oracle (forward + backward) on a bounded sample of neurons, on one
    host core.

    Returns (neuron-steps/s, description of the sample, neuron-steps timed, seconds, core)."""
    import oracle
    oracle.build()
    ocfg = oracle.OracleConfig(T=w.T, K=w.K, G=w.G, C=w.C, psi=w.psi, reset=w.reset,
                               theta=w.theta, beta=w.beta, stateless=w.stateless,
                               residual=w.residual, detach_reset=w.detach_reset)

    def run(M):
        x, chan, mrow, prm, mask, gs = inp_cpu_fn(M)
        t = time.perf_counter()
        oracle.forward(ocfg, x, chan, mrow, *prm, mask)
        oracle.backward(ocfg, x, chan, mrow, *prm, mask, gs)
        return time.perf_counter() - t

    with pinned_to_one_core() as core:
        M = 256
        dt = run(M)
        while dt < 0.3 and M < w.B * w.N:
            M = min(M * 4, w.B * w.N)
            dt = run(M)
        M = int(min(w.B * w.N, max(1, M * target_s / max(dt, 1e-6))))
        dt = run(M)
    ns = M * w.T
    return (ns / dt, f"{M} neurons x T={w.T} of the {w.name} layer (forward + backward), "
            f"1 thread", ns, dt, core)


def cpu_inputs_from(w, inp):
    """Sampler of M neurons of the device-resident inputs, as host arrays for the oracle."""
    import numpy as np
    import torch

    def fn(M):
        M = min(M, w.B * w.N)
        flat = torch.arange(M, device=inp["x"].device) * ((w.B * w.N) // M)
        b, n = flat // w.N, flat % w.N
        if w.layout == "paper":                 # [T, B, N/inner, K, inner] -> [T, M, K]
            x5 = inp["x"].reshape(w.T, w.B, w.N // w.inner, w.K, w.inner)
            x = x5[:, b, n // w.inner, :, n % w.inner].transpose(0, 1).cpu()
        else:
            x = inp["x"][:, b, n, :].cpu()
        gs = inp["gs"][:, b, n].cpu()
        nn = n.cpu().numpy()
        chan = ((nn // w.inner) % w.C).astype(np.int32)
        mrow = (nn if w.mask_per_neuron else chan).astype(np.int32)
        prm = [inp[k].cpu() for k in ("alpha", "xi", "zeta", "kappa")]
        mask = None if inp["mask"] is None else inp["mask"].cpu()
        return x, chan, mrow, prm, mask, gs
    return fn


def cpu_baseline_block(w, inp, target_s):
    rate, sample, _, dt, core = oracle_sample_rate(w, cpu_inputs_from(w, inp), target_s)
    return {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": sample + f", {dt:.1f} s", "pinned_core": core,
            "cpu_model": host_cpu_model(), "host_cpus": os.cpu_count()}


# ------------------------------------------------------------------ arms
def workload_of(args, name=None):
    from paper_2412_06355_gb300.workloads import WORKLOADS
    w = WORKLOADS[name or args.workload]
    if args.psi:
        w = w.with_(psi=args.psi)
    if args.batch:
        w = w.with_(B=args.batch)
    if args.variant != "stateful":
        w = w.with_(stateless=args.variant in ("stateless", "resstateless"),
                    residual=args.variant.startswith("res"))
    return w


def block_names(args):
    """The layer workloads reported as blocks beside the headline."""
    if args.blocks is None:
        return list(BLOCKS) if args.workload == HEADLINE and not args.batch else []
    if args.blocks.strip().lower() in ("", "none"):
        return []
    return [b.strip() for b in args.blocks.split(",") if b.strip() and b.strip() != args.workload]


def config_dict(w, extra=None):
    d = {"workload": w.name, "T": w.T, "B": w.B, "N": w.N, "K": w.K, "G": w.G, "C": w.C,
         "inner": w.inner, "x_dtype": w.dtype, "state_dtype": "f32", "psi": w.psi,
         "reset": w.reset,
         "mask": (None if w.mask_p is None else
                  f"Bernoulli({w.mask_p}) per {'neuron' if w.mask_per_neuron else 'channel'}"),
         "x_density": w.x_density, "layout": w.layout,
         "variant": ("res" if w.residual else "") + ("stateless" if w.stateless else "stateful")}
    if extra:
        d.update(extra)
    return d


def dtype_label(w) -> str:
    """The arithmetic type of the path: state and arithmetic are float32 for every layer;
    the tensors in HBM are float32 or bfloat16."""
    return "f32" if w.dtype == "f32" else "f32 (bf16 inputs/outputs, f32 state)"


def slice_workload(w, M):
    """The same layer kind with about M neurons (neurons are independent: the
    per-neuron work is unchanged). Whole rows of C*inner neurons are kept; below one
    row the channel count shrinks."""
    P = w.C * w.inner
    if M >= P:
        rows = max(1, min(M // P, w.N // P))
        return w.with_(B=1, N=rows * P)
    c = max(1, M // w.inner)
    return w.with_(B=1, C=c, N=c * w.inner)


def run_reference(args):
    """The oracle, as it stands, on the host cores: the slow baseline arm."""
    if int(os.environ.get("RANK", "0")) != 0:
        return
    import oracle
    from paper_2412_06355_gb300 import workloads
    oracle.build()
    w = workload_of(args)

    def one_step(ws, inp):
        oracle.forward_layer(ws, inp)
        oracle.backward_layer(ws, inp)

    # size one step to about 90 s / (steps + warmup), between 0.2 s and 2 s
    per_step = max(0.2, min(2.0, 90.0 / max(args.steps + args.warmup, 1)))
    with pinned_to_one_core() as core:
        probe = slice_workload(w, 4096)
        pin = workloads.make_inputs(probe, "cpu")
        t = time.perf_counter()
        one_step(probe, pin)
        rate = probe.neuron_steps / max(time.perf_counter() - t, 1e-6)
        ws = slice_workload(w, int(rate * per_step / w.T))
        inp = workloads.make_inputs(ws, "cpu")
        for _ in range(args.warmup):
            one_step(ws, inp)
        t = time.perf_counter()
        for _ in range(args.steps):
            one_step(ws, inp)
        dt = time.perf_counter() - t
    value = args.steps * ws.neuron_steps / dt
    sample = (f"{ws.B * ws.N} neurons x T={w.T} per step ({ws.C} channels x {ws.inner}; a "
              f"slice of the {w.name} layer), float64 forward + backward, 1 thread")
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * dt / max(args.steps, 1), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference",
            "config": config_dict(w, {"sample_neurons_per_step": ws.B * ws.N}),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": sample, "pinned_core": core,
                             "cpu_model": host_cpu_model(), "host_cpus": os.cpu_count()},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def time_lif(T, B, N, dtype, steps, warmup, stream):
    """Fused LIF layer fwd+bwd (the point-neuron baseline) timed like the DendSN step."""
    import torch
    from paper_2412_06355_gb300 import binding, workloads
    inp = workloads.make_lif_inputs(T, B, N, dtype, seed=11, device="cuda")
    cfg = binding.make_lif_config(T, B, N, dtype)
    x, gs = inp["x"], inp["gs"]
    saved = binding.lif_workspace(cfg)
    spikes, gx = torch.empty_like(x), torch.empty_like(x)

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        binding.dendsn_lif_forward(cfg, x, spikes, None, saved, stream)
        if ev is not None:
            ev[1].record(stream)
        binding.dendsn_lif_backward(cfg, x, gs, None, saved, gx, stream)
        if ev is not None:
            ev[2].record(stream)

    for _ in range(warmup):
        step()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    torch.cuda.synchronize()
    for i in range(steps):
        step(ev[i])
    torch.cuda.synchronize()
    fwd = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    bwd = statistics.mean(e[1].elapsed_time(e[2]) for e in ev)
    ms = fwd + bwd
    sx = x.element_size()
    nbytes = T * B * N * 5 * sx            # fwd: x + S; bwd: x + gS + gX
    return {"T": T, "B": B, "N": N, "x_dtype": dtype, "ms_per_step": ms, "forward_ms": fwd,
            "backward_ms": bwd, "value": T * B * N / (ms / 1e3), "unit": UNIT,
            "algorithmic_bytes_per_step": nbytes, "gbs": nbytes / (ms / 1e3) / 1e9}


class Layer:
    """One layer workload resident on the device: inputs, outputs, workspaces and the
    forward / backward calls of one step through the C ABI."""

    def __init__(self, w, args, dev, rank, stream):
        import torch
        from paper_2412_06355_gb300 import binding, distributed, workloads
        self.w, self.args, self.stream = w, args, stream
        self.w_rank = w.with_(seed=w.seed + 1000 * rank)
        self.cfg = binding.config_of(w)
        self.inp = workloads.make_inputs(self.w_rank, str(dev))
        inp = self.inp
        self.x, self.gs = inp["x"], inp["gs"]
        self.prm = [inp[k] for k in ("alpha", "xi", "zeta", "kappa")]
        self.mask = inp["mask"]
        self.saved, self.scratch = binding.workspace(self.cfg, dev)
        self.spikes = torch.empty((w.T, w.B, w.N), dtype=self.x.dtype, device=dev)
        self.gx = torch.empty_like(self.x)
        self.grads, views = distributed.param_grad_buffer(w.C, w.K, w.Kb, dev,
                                                          with_beta=args.plif)
        self.gviews = [views[k] for k in ("galpha", "gxi", "gzeta", "gkappa")]
        self.gbeta = views.get("gbeta")
        self.graphs = None
        self.launches_per_step = None

    def fwd(self, strm):
        from paper_2412_06355_gb300 import binding
        if self.graphs is not None:
            return self.graphs[0].replay()
        binding.dendsn_forward(self.cfg, self.x, *self.prm, self.mask, self.spikes, None,
                               self.saved, strm)

    def bwd(self, strm):
        from paper_2412_06355_gb300 import binding
        if self.graphs is not None:
            return self.graphs[1].replay()
        if self.args.plif:
            binding.dendsn_backward_plif(self.cfg, self.x, *self.prm, self.mask, self.gs, None,
                                         self.saved, self.gx, *self.gviews, self.gbeta,
                                         self.scratch, strm)
        else:
            binding.dendsn_backward(self.cfg, self.x, *self.prm, self.mask, self.gs, None,
                                    self.saved, self.gx, *self.gviews, self.scratch, strm)

    def capture(self):
        """--graph: the forward and the backward each captured into a CUDA graph once, then
        replayed every step (no per-step host launch work)."""
        import torch
        from paper_2412_06355_gb300 import binding
        side = torch.cuda.Stream()
        side.wait_stream(self.stream)
        with torch.cuda.stream(side):               # one eager step before capturing
            self.fwd(side)
            self.bwd(side)
        self.stream.wait_stream(side)
        torch.cuda.synchronize()
        n0 = binding.launch_count()
        graphs = []
        for part in (self.fwd, self.bwd):
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr):
                part(torch.cuda.current_stream())
            graphs.append(gr)
        self.launches_per_step = binding.launch_count() - n0
        self.graphs = graphs


def time_layer(layer, args, world, dev):
    """Warm-up, then args.steps steps with an event pair around each step's forward and
    backward (the split), then exactly args.steps timed steps without them, between
    barriers and synchronizes: the layer's time. Each event record is a stream operation of
    its own (about 2 us between two kernels, 6 us a step), instrumentation that a training
    step does not have. Returns the per-step event times, the whole-region time of the plain
    pass (max over ranks; and that of the instrumented pass), its wall-clock window and its
    launch count."""
    import torch
    import torch.distributed as dist
    from paper_2412_06355_gb300 import binding, distributed
    stream = layer.stream

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        layer.fwd(stream)
        if ev is not None:
            ev[1].record(stream)
        layer.bwd(stream)
        if ev is not None:
            ev[2].record(stream)
        if world > 1:
            distributed.sum_param_grads(layer.grads)

    for _ in range(args.warmup):
        step()
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    start.record(stream)
    for i in range(args.steps):
        step(ev[i])
    end.record(stream)
    torch.cuda.synchronize()
    ms_events = start.elapsed_time(end)

    # the timed region: the same steps without the per-step event records
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    n_launch0 = binding.launch_count()
    t0 = time.time()
    start.record(stream)
    for i in range(args.steps):
        step()
    end.record(stream)
    torch.cuda.synchronize()
    t1 = time.time()
    n_launch = binding.launch_count() - n_launch0
    if layer.launches_per_step is not None:         # replays launch without library calls
        n_launch = layer.launches_per_step * args.steps
    if world > 1:
        dist.barrier()
    ms = start.elapsed_time(end)
    if world > 1:
        t = torch.tensor([ms, ms_events], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms, ms_events = float(t[0].item()), float(t[1].item())
    return dict(ms=ms, ms_events=ms_events, fwd_ms=[e[0].elapsed_time(e[1]) for e in ev],
                bwd_ms=[e[1].elapsed_time(e[2]) for e in ev], t0=t0, t1=t1, launches=n_launch)


def time_e2e(layer, args, world, dev):
    """End to end through the C ABI from pinned host buffers, copies inside the timed region.

    Each step is the headline call itself (one forward and one backward over the whole
    batch) between a host->device copy of its inputs (x, dL/dS) and a device->host copy of
    its result, the parameter gradients (what a training step hands to the optimizer; the
    spikes and dL/dX are the tensors the next and the previous layer read on the device).
    Two sets of device buffers alternate between steps, and the copies of each direction and
    the kernels run on three streams ordered by events, so the next step's upload overlaps
    this step's kernels and download. The host waits for each step's result before it
    enqueues the step after next. Timed on the wall clock."""
    import torch
    import torch.distributed as dist
    from paper_2412_06355_gb300 import binding, distributed
    w, x, gs, cfg = layer.w, layer.x, layer.gs, layer.cfg
    alpha, xi, zeta, kappa = layer.prm
    mask = layer.mask
    pin = dict(pin_memory=True)
    x_h = torch.empty(x.shape, dtype=x.dtype, **pin)
    gs_h = torch.empty(gs.shape, dtype=gs.dtype, **pin)
    x_h.copy_(x)
    gs_h.copy_(gs)
    ng = layer.grads.numel()
    g_h = torch.empty(ng, dtype=torch.float32, **pin)
    sets = []
    for _ in range(2):
        g_d = torch.empty(ng, dtype=torch.float32, device=dev)
        sets.append(dict(x=torch.empty_like(x), gs=torch.empty_like(gs),
                         s=torch.empty((w.T, w.B, w.N), dtype=x.dtype, device=dev),
                         gx=torch.empty_like(x), ws=binding.workspace(cfg, dev), g=g_d,
                         gv=distributed.split_param_grads(g_d, w.C, w.K, w.Kb)))
    h2d = x_h.numel() * x_h.element_size() + gs_h.numel() * gs_h.element_size()
    d2h = g_h.numel() * g_h.element_size()
    up, comp, down = torch.cuda.Stream(), torch.cuda.Stream(), torch.cuda.Stream()
    ev = lambda: torch.cuda.Event()                   # noqa: E731
    loaded, computed, returned = ([ev(), ev()] for _ in range(3))

    def e2e_step(k):
        i = k % 2
        d = sets[i]
        saved, scratch = d["ws"]
        with torch.cuda.stream(up):
            up.wait_event(computed[i])               # the step before last has read set i
            d["x"].copy_(x_h, non_blocking=True)
            d["gs"].copy_(gs_h, non_blocking=True)
            loaded[i].record(up)
        comp.wait_event(loaded[i])
        comp.wait_event(returned[i])                 # set i's results of two steps ago are home
        binding.dendsn_forward(cfg, d["x"], alpha, xi, zeta, kappa, mask, d["s"], None, saved,
                               comp)
        binding.dendsn_backward(cfg, d["x"], alpha, xi, zeta, kappa, mask, d["gs"], None, saved,
                                d["gx"], *d["gv"], scratch, comp)
        if world > 1:
            with torch.cuda.stream(comp):
                dist.all_reduce(d["g"])              # the data-parallel gradient sum
        computed[i].record(comp)
        with torch.cuda.stream(down):
            down.wait_event(computed[i])
            g_h.copy_(d["g"], non_blocking=True)
            returned[i].record(down)

    ke = max(3, min(args.steps, 20))
    for k in range(3):
        e2e_step(k)
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for k in range(ke):
        e2e_step(k)
        if k > 0:
            returned[(k - 1) % 2].synchronize()      # the previous step's results are on the host
    torch.cuda.synchronize()
    ems = (time.perf_counter() - t0) * 1e3
    assert bool(torch.isfinite(g_h).all())
    if world > 1:
        t = torch.tensor([ems], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ems = float(t.item())
    return {"value": world * ke * w.neuron_steps / (ems / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "steps": ke,
            "ms_per_step": ems / ke, "streams": 3,
            "timing": "wall clock, host waits for each step's result (the parameter gradients)",
            "launch_geometry": f"the headline call (one forward and one backward of B={w.B}), "
                               "two device buffer sets alternating"}


def layer_report(layer, timing, world, dev, peak, peak_kind, clock):
    """Roofline of the dominant kernel, the step's HBM fraction and the throughput of one
    layer from its timing."""
    import torch
    w = layer.w
    ab = w.algorithmic_bytes()
    ops = w.fp32_ops_per_neuron_step()
    fwd_avg, bwd_avg = statistics.mean(timing["fwd_ms"]), statistics.mean(timing["bwd_ms"])
    fname, bname = kernel_names(w)
    if bwd_avg >= fwd_avg:
        kname, kbytes, kms, kops = bname, ab["backward"], bwd_avg, ops["backward"]
    else:
        kname, kbytes, kms, kops = fname, ab["forward"], fwd_avg, ops["forward"]
    achieved = kbytes / (kms / 1e3) / 1e9
    # the float32 roof of the same kernel: its float32 operations (a cost model counted from
    # the equations) against SMs x 128 FMA lanes x the SM clock
    sm_mhz = (clock or {}).get("sm_max_mhz") or NOMINAL_SM_MHZ
    fp32_peak = (torch.cuda.get_device_properties(dev).multi_processor_count *
                 FP32_LANES_PER_SM * sm_mhz * 1e6)
    ops_launch = kops * w.neuron_steps
    t_hbm, t_alu = kbytes / (peak * 1e9), ops_launch / fp32_peak
    alu = {"fp32_ops_per_neuron_step": kops, "fp32_ops_per_launch": ops_launch,
           "achieved_tops": ops_launch / (kms / 1e3) / 1e12, "peak_tops": fp32_peak / 1e12,
           "frac": ops_launch / (kms / 1e3) / fp32_peak,
           "peak_basis": f"SMs x {FP32_LANES_PER_SM} FP32 lanes x {sm_mhz:.0f} MHz",
           "min_ms_at_fp32_peak": t_alu * 1e3, "min_ms_at_hbm_peak": t_hbm * 1e3}
    step_ms = timing["ms"] / layer.args.steps
    value = world * w.neuron_steps / (step_ms / 1e3)
    ab_unit = kbytes / w.neuron_steps
    roof = {**({"bound": "hbm", "kernel": kname, "achieved": achieved, "peak": peak,
                "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak}
               if t_hbm >= t_alu else
               {"bound": "alu", "kernel": kname, "achieved": alu["achieved_tops"],
                "peak": alu["peak_tops"], "peak_kind": alu["peak_basis"],
                "unit": "FP32 Top/s", "frac": alu["frac"]}),
            "hbm_frac": achieved / peak,
            "frac_of_8tbs": achieved / NOMINAL_HBM_GBS,
            "alu": alu,
            # counters were taken on the plain backward build, not the dL/dbeta one
            "traffic": None if layer.args.plif else recorded_traffic(kname, w.name),
            "algorithmic_bytes_per_neuron_step": ab_unit,
            "neuron_steps_per_launch": w.neuron_steps,
            "algorithmic_bytes_per_launch": kbytes, "avg_launch_ms": kms}
    hbm = {"algorithmic_bytes_per_step": ab["total"],
           "step_gbs": ab["total"] / (step_ms / 1e3) / 1e9,
           "frac_of_8tbs": ab["total"] / (step_ms / 1e3) / 1e9 / NOMINAL_HBM_GBS,
           "frac_of_measured": ab["total"] / (step_ms / 1e3) / 1e9 / peak,
           "forward_ms": fwd_avg, "backward_ms": bwd_avg,
           "step_ms_with_step_events": timing["ms_events"] / layer.args.steps}
    return value, step_ms, roof, hbm


def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_2412_06355_gb300 import binding

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        torch.cuda.set_device(0)
    if args.graph and world > 1:
        raise SystemExit("--graph times one GPU")
    dev = torch.device("cuda", torch.cuda.current_device())
    binding.load()
    stream = torch.cuda.current_stream()
    peak, peak_kind = measured_hbm_peak()
    clocks = ClockSampler(dev.index)
    if rank == 0:
        clocks.start()

    names = [args.workload] + block_names(args)
    results = []                                     # (layer workload, timing, e2e)
    e2e = None
    for i, name in enumerate(names):
        w = workload_of(args, name)
        layer = Layer(w, args, dev, rank, stream)
        if args.graph:
            layer.capture()
        timing = time_layer(layer, args, world, dev)
        if i == 0 and not args.no_e2e:
            e2e = time_e2e(layer, args, world, dev)
        cpu = None
        results.append([layer, timing, cpu])
        log(f"{name}: {timing['ms'] / args.steps:.4f} ms per step")
        if i > 0:
            # the layer's device buffers go before the next one is drawn; the host-side CPU
            # baseline sample is drawn from the inputs later, so keep only what it needs
            layer.saved = layer.scratch = layer.spikes = layer.gx = None
    clock_rows = clocks.stop() if rank == 0 else []

    lif = None
    if rank == 0 and not args.no_lif:
        # the paper compares DendSN with LIF layers (Results, efficiency paragraph): here a
        # LIF layer with the same neurons as the conv layer (one current each), and one fed
        # the same input tensor (N*K point neurons)
        wl = next((r[0].w for r in results if r[0].w.name == "conv"), results[0][0].w)
        lay = next(r for r in results if r[0].w is wl)
        steps_l = max(3, min(args.steps, 50))
        same_n = time_lif(wl.T, wl.B, wl.N, wl.dtype, steps_l, 3, stream)
        same_x = time_lif(wl.T, wl.B, wl.N * wl.K, wl.dtype, steps_l, 3, stream)
        for d in (same_n, same_x):
            d["frac_of_measured"] = d["gbs"] / peak
        step_ms_l = lay[1]["ms"] / args.steps
        lif = {"workload": wl.name, "same_neurons": same_n, "same_input": same_x,
               "dendsn_over_lif_same_neurons": (wl.neuron_steps / (step_ms_l / 1e3)) /
                                               same_n["value"],
               "dendsn_over_lif_same_input": same_x["ms_per_step"] / step_ms_l,
               "note": "layer-level ratios of fwd+bwd throughput; the paper's 0.92 is for "
                       "whole networks (Tiny ImageNet VGG, Triton kernels)"}

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # CPU baselines last: the oracle runs pinned to one host core after all GPU timing
    blocks = []
    head = None
    for i, (layer, timing, _) in enumerate(results):
        w = layer.w
        clock = ClockSampler.summarize(clock_rows, timing["t0"], timing["t1"])
        value, step_ms, roof, hbm = layer_report(layer, timing, world, dev, peak, peak_kind,
                                                 clock)
        cpu = None
        if not args.no_cpu_baseline and world == 1:
            cpu = cpu_baseline_block(w, layer.inp, args.cpu_seconds)
        x_bytes = layer.x.numel() * layer.x.element_size()
        cfg = config_dict(w, {
            "l2": f"inputs larger than L2: x is {x_bytes / 2**20:.0f} MiB per step "
                  f"(L2 {L2_BYTES // 2**20} MiB), no flush",
            "parallelism": f"dp{world}" if world > 1 else "single GPU",
            "soma": "plif (learnable beta)" if args.plif else "lif",
            "launch": "cuda graph replay" if args.graph else "eager"})
        block = {"workload": w.name, "value": value, "unit": UNIT, "ms_per_step": step_ms,
                 "forward_ms": hbm["forward_ms"], "backward_ms": hbm["backward_ms"],
                 "dtype": dtype_label(w), "config": cfg, "roofline": roof, "hbm": hbm,
                 "clocks": clock, "gpu_launches": timing["launches"], "cpu_baseline": cpu}
        if i == 0:
            head = block
        else:
            blocks.append(block)

    line = {
        "metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": head["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": head["dtype"], "data": "synthetic", "config": head["config"],
        "roofline": head["roofline"], "hbm": head["hbm"], "clocks": head["clocks"],
        "e2e": e2e, "gpu_launches": head["gpu_launches"], "cpu_baseline": head["cpu_baseline"],
        "blocks": blocks, "lif_baseline": lif,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
