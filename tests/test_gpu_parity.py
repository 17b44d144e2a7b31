"""GPU parity: the CUDA path through the C ABI against the float64 oracle.

Tolerances and the handling of threshold-ambiguous steps are in tests/parity.py.
* every layer workload at a size the oracle finishes in seconds (all neurons),
  with both branch nonlinearities;
* edge cases: every compiled (K, G), ragged tiles and chunks, T = 0 / 1,
  empty batch, every flag, extreme threshold/decay;
* the full-size workloads in the benchmark's launch configuration, compared on a
  sample of neurons (neurons are independent), with parameter gradients checked
  by giving the non-sampled neurons zero upstream gradient (the backward is
  linear in it, so the sums then run over the sample only).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2412_06355_gb300 import binding, workloads
from paper_2412_06355_gb300.workloads import WORKLOADS, scaled

from parity import (BF16_ATOL_REL, BF16_RTOL, G_ATOL_REL, G_RTOL, GX_ATOL_REL, P_ATOL_REL,
                    V_ATOL, V_RTOL, assert_close, check_layer, direction_rounding_allowance,
                    first_ambiguous_step, gx_atol_rel, needs_allowance,
                    soma_rounding_allowance, to_dev)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("these tests need a CUDA device")
    binding.load()
    oracle.build()


SCALED = {
    "tiny": WORKLOADS["tiny"],
    "conv": scaled(WORKLOADS["conv"], B=2),
    "deepconv_bf16": scaled(WORKLOADS["deepconv_bf16"], B=2),
    "event": WORKLOADS["event"].with_(C=32, N=32 * 1024, B=2),
    "token_dbg": scaled(WORKLOADS["token_dbg"], B=2),
    "conv_paper_p4b2": scaled(WORKLOADS["conv_paper_p4b2"], B=2),
    "deepconv_bf16_paper": scaled(WORKLOADS["deepconv_bf16"], B=2).with_(layout="paper"),
    "l5pc": WORKLOADS["l5pc"],
    "long_t": WORKLOADS["long_t"].with_(B=1, N=1024, C=1),
}


@pytest.mark.parametrize("psi", ["mh", "identity"])
@pytest.mark.parametrize("name", list(SCALED))
def test_layer_workloads(name, psi):
    w = SCALED[name].with_(psi=psi)
    info = check_layer(w)
    assert info["spikes"] > 0.0


KG = [(1, 1), (2, 1), (2, 2), (4, 1), (4, 2), (4, 4), (8, 1), (8, 2), (8, 4),
      (16, 1), (16, 2), (16, 4)]


@pytest.mark.parametrize("layout", ["kinner", "paper"])
@pytest.mark.parametrize("K,G", KG)
def test_every_compiled_kg(K, G, layout):
    i = KG.index((K, G))
    w = workloads.Workload(
        f"kg{K}_{G}", T=9, B=3, N=35 * 2, K=K, G=G, C=5, inner=7,
        dtype="bf16" if i % 3 == 2 else "f32", psi="mh" if i % 2 == 0 else "identity",
        reset="soft" if i % 4 == 1 else "hard", mask_p=0.6 if i % 2 else None,
        mask_per_neuron=(i % 4 == 3), layout=layout, seed=100 + i)
    check_layer(w)


@pytest.mark.parametrize("inner", [40, 64])      # 64: the forward stages inputs per warp
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("K,G,T", [(2, 2, 3), (4, 2, 4), (4, 1, 12), (8, 1, 4), (8, 1, 8),
                                   (8, 2, 9), (16, 4, 5)])
def test_paper_layout_is_bitwise_the_kinner_layer(K, G, T, dtype, inner):
    """Only the addresses differ between the layouts: every output must be bit-identical."""
    w = workloads.Workload("lay", T=T, B=3, N=4 * 2 * inner, K=K, G=G, C=4, inner=inner,
                           dtype=dtype, psi="mh", reset="hard", mask_p=0.7, seed=21)
    wp = w.with_(layout="paper")
    outs = []
    for ww in (w, wp):
        inp = to_dev(workloads.make_inputs(ww, "cpu", with_gv=True))
        cfg = binding.config_of(ww)
        saved, scratch = binding.workspace(cfg)
        s, v = binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                               inp["kappa"], inp["mask"], want_v=True, saved=saved)
        g = binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                             inp["kappa"], inp["mask"], inp["gs"], inp["gv"], saved, scratch,
                             want_beta=True)
        outs.append((s, v, g))
    torch.cuda.synchronize()
    (s, v, g), (sp, vp, gp) = outs
    assert torch.equal(s, sp) and torch.equal(v, vp)
    assert torch.equal(g["gx"], workloads.from_paper_layout(gp["gx"], w.N, w.K, w.inner))
    for k in ("galpha", "gxi", "gzeta", "gkappa", "gbeta"):
        assert torch.equal(g[k], gp[k]), k


@pytest.mark.parametrize("kw", [
    dict(stateless=True), dict(residual=True), dict(stateless=True, residual=True),
    dict(detach_reset=True), dict(detach_reset=True, reset="soft"),
    dict(reset="soft", psi="identity"), dict(theta=0.0), dict(beta=0.0),
    dict(theta=0.25, beta=0.95), dict(mask_p=0.5), dict(mask_p=0.5, mask_per_neuron=True),
    dict(mask_p=0.0),
], ids=lambda kw: "-".join(f"{k}={v}" for k, v in kw.items()))
def test_variants(kw):
    w = workloads.Workload("var", T=6, B=4, N=4 * 96, K=8, G=1, C=4, inner=96, dtype="f32",
                           psi="mh", reset="hard", seed=7).with_(**kw)
    check_layer(w)


@pytest.mark.parametrize("T", [4, 8])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kw", [
    dict(), dict(mask_p=0.5, mask_per_neuron=True), dict(mask_p=0.5),
    dict(reset="soft", psi="identity"), dict(detach_reset=True), dict(stateless=True),
    dict(residual=True), dict(layout="paper"),
], ids=lambda kw: "-".join(f"{k}={v}" for k, v in kw.items()) or "plain")
def test_one_chunk_rows_of_8_compartments(kw, dtype, T):
    # rows of one full chunk of 8-compartment neurons: the phased backward (bf16, or T == 8),
    # and for float32 T == 4 the two-rows-per-thread backward of split lanes; B = 5 gives
    # threads odd row counts (the unpaired last row); the residual variant takes the
    # chunked kernel
    w = workloads.Workload("onechunk", T=T, B=5, N=3 * 128, K=8, G=1, C=3, inner=128,
                           dtype=dtype, psi="mh", reset="hard", seed=41).with_(**kw)
    check_layer(w)


def test_phased_backward_grad_spike_paths_are_bitwise_equal():
    """The phased backward takes dL/dS into shared memory by 4-byte cp.async words when gs
    is 4-byte aligned and B*N is even, else into registers: both paths give the same bits,
    and a layer with odd B*N (register path) matches the oracle."""
    w = workloads.Workload("gsp", T=8, B=5, N=3 * 128, K=8, G=1, C=3, inner=128, dtype="bf16",
                           psi="mh", reset="soft", mask_p=0.5, seed=43)
    inp = to_dev(workloads.make_inputs(w, "cpu", with_gv=True))
    cfg = binding.config_of(w)
    prm = [inp[k] for k in ("alpha", "xi", "zeta", "kappa")]
    for want_beta in (False, True):
        outs = []
        for off in (0, 1):                   # element offset 1: gs only 2-byte aligned
            buf = torch.zeros(inp["gs"].numel() + 1, dtype=inp["gs"].dtype, device="cuda")
            gs = buf[off:off + inp["gs"].numel()].view(inp["gs"].shape)
            gs.copy_(inp["gs"])
            saved, scratch = binding.workspace(cfg)
            binding.forward(cfg, inp["x"], *prm, inp["mask"], want_v=False, saved=saved)
            outs.append(binding.backward(cfg, inp["x"], *prm, inp["mask"], gs, inp["gv"], saved,
                                         scratch, want_beta=want_beta))
        torch.cuda.synchronize()
        for k in outs[0]:
            assert torch.equal(outs[0][k], outs[1][k]), (k, want_beta)
    check_layer(w.with_(N=3 * 45, inner=45, seed=44))      # B*N = 675


@pytest.mark.parametrize("T", [1, 2, 3, 5, 8, 9, 16, 17, 64, 70])
def test_time_lengths_and_checkpoint_chunks(T):
    w = workloads.Workload("t", T=T, B=3, N=2 * 160, K=4, G=2, C=2, inner=160, dtype="f32",
                           psi="identity" if T % 2 else "mh", reset="hard" if T % 3 else "soft",
                           x_mean=0.5, seed=T)
    check_layer(w)


@pytest.mark.parametrize("T", [5, 9, 13])
def test_several_rows_per_thread_with_ragged_time(T):
    # 640 rows of 1024 neurons: each thread walks R > 1 rows, so the prefetch of the
    # next row crosses a ragged last chunk (T not a multiple of the load batch / chunk)
    w = workloads.Workload("rows", T=T, B=640, N=1024, K=4, G=1, C=2, inner=512, dtype="f32",
                           psi="mh", reset="hard", seed=30 + T)
    check_layer(w, with_gv=False)


def test_ragged_column_tiles_and_odd_inner():
    # P = C*inner = 300: not a multiple of any tile width; inner = 100 is not a power of 2
    w = workloads.Workload("ragged", T=5, B=3, N=600, K=4, G=1, C=3, inner=100, dtype="f32",
                           psi="mh", reset="hard", seed=9)
    check_layer(w)
    w = w.with_(K=8, dtype="bf16", inner=50, N=300, seed=10)
    check_layer(w)


def test_large_inner_and_sparse_zero_inputs():
    # exact zeros with xi = 0 hit r_b = 0 (subgradient 0) for the identity branch
    w = workloads.Workload("zeros", T=12, B=2, N=2048, K=4, G=2, C=2, inner=1024, dtype="f32",
                           psi="identity", reset="hard", x_mean=0.8, x_density=0.2, seed=12)
    inp = workloads.make_inputs(w, "cpu", with_gv=True)
    inp["xi"].zero_()
    check_layer(w, seed_inputs=inp)


def test_empty_shapes():
    for T, B in ((0, 2), (3, 0)):
        w = workloads.Workload("empty", T=T, B=B, N=64, K=4, G=1, C=4, inner=16, dtype="f32",
                               psi="mh", reset="hard")
        cfg = binding.config_of(w)
        inp = to_dev(workloads.make_inputs(w, "cpu"))
        s, _ = binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"], None)
        g = binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"], None,
                             inp["gs"], None, want_beta=True)
        torch.cuda.synchronize()
        assert s.numel() == 0
        for k in ("galpha", "gxi", "gzeta", "gkappa", "gbeta"):
            assert torch.count_nonzero(g[k]).item() == 0


def test_backward_is_deterministic():
    w = scaled(WORKLOADS["token_dbg"], B=2)
    inp = to_dev(workloads.make_inputs(w, "cpu"))
    cfg = binding.config_of(w)
    outs = []
    for _ in range(2):
        saved, scratch = binding.workspace(cfg)
        binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"],
                        inp["mask"], saved=saved)
        outs.append(binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                                     inp["kappa"], inp["mask"], inp["gs"], None, saved, scratch,
                                     want_beta=True))
    for k in outs[0]:
        assert torch.equal(outs[0][k], outs[1][k]), k


def test_misaligned_device_pointer_is_rejected():
    w = workloads.Workload("a", T=4, B=1, N=64, K=4, G=1, C=4, inner=16, dtype="f32",
                           psi="mh", reset="hard")
    cfg = binding.config_of(w)
    inp = to_dev(workloads.make_inputs(w, "cpu"))
    buf = torch.empty(inp["x"].numel() + 1, dtype=torch.float32, device="cuda")
    x_off = buf[1:].view(inp["x"].shape)            # 4-byte offset: not 16-byte aligned
    with pytest.raises(binding.DendSNError) as e:
        binding.forward(cfg, x_off, inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"], None)
    assert e.value.status == 3


def test_autograd_function_layer_wide_alpha():
    """DendSNFunction with the paper's scalar alpha: gradient = sum of the [C,K] one."""
    w = workloads.Workload("ag", T=4, B=2, N=128, K=4, G=2, C=4, inner=32, dtype="f32",
                           psi="mh", reset="hard", seed=21)
    inp = to_dev(workloads.make_inputs(w, "cpu"))
    cfg = binding.config_of(w)
    x = inp["x"].clone().requires_grad_(True)
    alpha = torch.tensor(0.7, device="cuda", requires_grad=True)
    xi = inp["xi"].clone().requires_grad_(True)
    zeta = inp["zeta"].clone().requires_grad_(True)
    kappa = inp["kappa"].clone().requires_grad_(True)
    s = binding.DendSNFunction.apply(x, alpha, xi, zeta, kappa, None, cfg)
    (s * inp["gs"]).sum().backward()
    full = inp["alpha"].clone().fill_(0.7)
    ref = binding.backward(cfg, inp["x"], full, inp["xi"], inp["zeta"], inp["kappa"], None,
                           inp["gs"], None, *binding.workspace(cfg))
    torch.cuda.synchronize()
    assert torch.allclose(alpha.grad, ref["galpha"].sum(), rtol=1e-5, atol=1e-6)
    assert torch.equal(x.grad, ref["gx"])
    assert torch.equal(kappa.grad, ref["gkappa"])


def test_autograd_function_learnable_beta():
    """A learnable somatic decay (PLIF soma) through autograd: its gradient is the sum of the
    per-channel dL/dbeta, checked against the float64 oracle."""
    w = workloads.Workload("plif", T=6, B=2, N=128, K=4, G=2, C=4, inner=32, dtype="f32",
                           psi="mh", reset="soft", beta=0.8, seed=23)
    inp = workloads.make_inputs(w, "cpu")
    dev = to_dev(inp)
    cfg = binding.config_of(w.with_(beta=0.5))          # the tensor's value must win
    beta = torch.tensor(0.8, device="cuda", requires_grad=True)
    x = dev["x"].clone().requires_grad_(True)
    s = binding.DendSNFunction.apply(x, dev["alpha"], dev["xi"], dev["zeta"], dev["kappa"],
                                     None, cfg, beta)
    s_o, v_o = oracle.forward_layer(w, inp)
    amb = torch.from_numpy(first_ambiguous_step(v_o, w.theta) < w.T)
    gs = inp["gs"].clone()
    gs[:, amb] = 0
    assert np.array_equal(oracle.to_f64(s)[:, ~amb.numpy()], s_o[:, ~amb.numpy()])
    (s * gs.cuda()).sum().backward()
    ref = oracle.backward_layer(w, inp, gs=gs)
    assert_close("dL/dbeta", [beta.grad.item()], [ref["gbeta"].sum()], G_RTOL, G_ATOL_REL,
                 atol_abs=1e-5 * float(np.sqrt(np.mean(ref["gbeta"] ** 2))))
    assert_close("grad_x", oracle.to_f64(x.grad), ref["gx"], G_RTOL, G_ATOL_REL)


# ------------------------------------------------------------------ full size, sampled
def sample_neurons(w, count, seed):
    rng = np.random.default_rng(seed)
    flat = rng.choice(w.B * w.N, size=min(count, w.B * w.N), replace=False)
    flat.sort()
    return flat // w.N, flat % w.N


def x_of_neurons(w, x, bt, nt):
    """[T, M, K] compartment values of neurons (bt[m], nt[m]) in either layout."""
    if w.layout == "paper":
        x5 = x.reshape(w.T, w.B, w.N // w.inner, w.K, w.inner)
        # separated advanced indices put the sample axis first: [M, T, K] -> [T, M, K]
        return x5[:, bt, nt // w.inner, :, nt % w.inner].transpose(0, 1)
    return x[:, bt, nt, :]


FULL = [(n, {}) for n in WORKLOADS] + [
    ("conv", dict(stateless=True, residual=True)),        # ResStateless (the Tiny ImageNet choice)
    ("conv", dict(stateless=True)),                       # Stateless (the CIFAR10-DVS choice)
    ("event", dict(residual=True, psi="identity")),       # ResStateful, identity branches
]


# element offsets beyond 2^31: T * B * N * K = 64 * 65 * 131072 * 4 = 2.18e9 (x alone 8.7 GB)
BIG = workloads.Workload("offsets_beyond_int32", T=64, B=65, N=131072, K=4, G=1, C=128,
                         inner=1024, dtype="f32", psi="mh", reset="hard", seed=41)


@pytest.mark.parametrize("name,kw", FULL + [("offsets_beyond_int32", {})],
                         ids=[n + "".join(f"-{k}" for k in kw) for n, kw in FULL] +
                         ["offsets_beyond_int32"])
def test_full_size_sampled(name, kw):
    w = (BIG if name == BIG.name else WORKLOADS[name]).with_(**kw)
    allow = needs_allowance(w)
    cfg = binding.config_of(w)
    inp = workloads.make_inputs(w, "cuda")          # full size, generated on the device
    b_idx, n_idx = sample_neurons(w, 3000, seed=w.seed)
    bt, nt = torch.from_numpy(b_idx).cuda(), torch.from_numpy(n_idx).cuda()

    # oracle on the sampled neurons (independent of the rest of the layer)
    xs = x_of_neurons(w, inp["x"], bt, nt).cpu()                       # [T, M, K]
    chan = ((n_idx // w.inner) % w.C).astype(np.int32)
    mrow = (n_idx if w.mask_per_neuron else chan).astype(np.int32)
    ocfg = oracle.OracleConfig(T=w.T, K=w.K, G=w.G, C=w.C, psi=w.psi, reset=w.reset,
                               theta=w.theta, beta=w.beta, stateless=w.stateless,
                               residual=w.residual)
    prm = [inp[k].cpu() for k in ("alpha", "xi", "zeta", "kappa")]
    mask = None if inp["mask"] is None else inp["mask"].cpu()
    s_o, v_o = oracle.forward(ocfg, xs, chan, mrow, *prm, mask)
    v_extra = (soma_rounding_allowance(w, oracle.to_f64(xs), chan, mrow, *prm, mask, v_o)
               if allow else 0.0)
    first = (first_ambiguous_step(v_o, w.theta, V_ATOL + V_RTOL * np.abs(v_o) + v_extra)
             if allow else first_ambiguous_step(v_o, w.theta))
    keep = first == w.T

    # upstream gradient: zero except on the unambiguous sampled neurons
    gs_sample = torch.zeros_like(inp["gs"])
    kb, kn = bt[torch.from_numpy(keep).cuda()], nt[torch.from_numpy(keep).cuda()]
    gs_sample[:, kb, kn] = inp["gs"][:, kb, kn]

    saved, scratch = binding.workspace(cfg)
    s, v = binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"],
                           inp["mask"], want_v=True, saved=saved)
    g = binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"],
                         inp["mask"], gs_sample, None, saved, scratch, want_beta=True)
    torch.cuda.synchronize()
    got_s = oracle.to_f64(s[:, bt, nt])
    got_v = oracle.to_f64(v[:, bt, nt])
    got_gx = oracle.to_f64(x_of_neurons(w, g["gx"], bt, nt))
    t_idx = np.arange(w.T)[:, None]
    assert_close("V^s", got_v, v_o, V_RTOL, 0.0, mask=t_idx <= first[None],
                 atol_abs=V_ATOL + v_extra)
    sm = t_idx < first[None]
    assert np.array_equal(got_s[sm], s_o[sm])

    ref = oracle.backward(ocfg, xs, chan, mrow, *prm, mask, gs_sample[:, bt, nt].cpu(),
                          want_dvs=True)
    rt = BF16_RTOL if w.dtype == "bf16" else G_RTOL
    if allow:
        extra = direction_rounding_allowance(w, oracle.to_f64(xs), chan, mrow, *prm, mask,
                                             ref["dvs"])
        ar = BF16_ATOL_REL if w.dtype == "bf16" else gx_atol_rel(w, inp["alpha"])
        p_rel = G_ATOL_REL
    else:
        extra, ar, p_rel = 0.0, GX_ATOL_REL, P_ATOL_REL
    assert_close("grad_x", got_gx, ref["gx"], rt, ar, atol_abs=extra)
    for k in ("galpha", "gxi", "gzeta", "gkappa", "gbeta"):
        assert_close(k, oracle.to_f64(g[k]), ref[k], G_RTOL, p_rel)
    # every non-sampled neuron received zero upstream gradient: its grad_x is zero
    gx = g["gx"]
    if w.layout == "paper":
        gx = workloads.from_paper_layout(gx, w.N, w.K, w.inner)
    gx_abs = gx.abs().sum(dim=(0, 3))
    gx_abs[bt, nt] = 0
    assert torch.count_nonzero(gx_abs).item() == 0


# ------------------------------------------------------------------ CUDA graphs
def test_cuda_graph_capture_and_replay():
    """A whole step (forward, backward, finalize) captured into a CUDA graph and replayed on
    new inputs written into the captured buffers gives the eager calls' bits."""
    w = workloads.Workload("graph", T=12, B=2, N=4 * 64, K=4, G=2, C=4, inner=64, dtype="f32",
                           psi="mh", reset="hard", mask_p=0.5, seed=51)
    cfg = binding.config_of(w)
    inp = to_dev(workloads.make_inputs(w, "cpu"))
    x, gs = inp["x"].clone(), inp["gs"].clone()
    p = [inp[k] for k in ("alpha", "xi", "zeta", "kappa")]
    saved, scratch = binding.workspace(cfg)
    spikes = torch.empty((w.T, w.B, w.N), device="cuda")
    gx = torch.empty_like(x)
    grads = [torch.empty_like(t) for t in p]

    def step(stream):
        binding.dendsn_forward(cfg, x, *p, inp["mask"], spikes, None, saved, stream)
        binding.dendsn_backward(cfg, x, *p, inp["mask"], gs, None, saved, gx, *grads, scratch,
                                stream)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step(side)                                    # warm-up outside the capture
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step(torch.cuda.current_stream())
    for seed in (52, 53):
        new = workloads.make_inputs(w.with_(seed=seed), "cpu")
        x.copy_(new["x"])
        gs.copy_(new["gs"])
        graph.replay()
        torch.cuda.synchronize()
        s_eager, _ = binding.forward(cfg, x, *p, inp["mask"], saved=binding.workspace(cfg)[0])
        sv, sc = binding.workspace(cfg)
        binding.forward(cfg, x, *p, inp["mask"], saved=sv)
        g = binding.backward(cfg, x, *p, inp["mask"], gs, None, sv, sc)
        torch.cuda.synchronize()
        assert torch.equal(spikes, s_eager)
        assert torch.equal(gx, g["gx"])
        for got, k in zip(grads, ("galpha", "gxi", "gzeta", "gkappa")):
            assert torch.equal(got, g[k]), k


def test_concurrent_streams_match_sequential_calls():
    """Two layers (one of them on the time-parallel kernels) run at the same time on two streams
    give the bits of running them one after the other: the library keeps no shared state."""
    ws = [workloads.Workload("cs_a", T=9, B=4, N=4 * 256, K=4, G=1, C=4, inner=256, dtype="f32",
                             psi="mh", reset="hard", mask_p=0.5, seed=61),
          workloads.Workload("cs_b", T=300, B=2, N=8 * 32, K=8, G=2, C=8, inner=32,
                             dtype="bf16", psi="identity", reset="soft", seed=62)]
    cfgs = [binding.config_of(w) for w in ws]
    inps = [to_dev(workloads.make_inputs(w, "cpu")) for w in ws]

    def run(k, stream):
        w, cfg, inp = ws[k], cfgs[k], inps[k]
        saved, scratch = binding.workspace(cfg)
        with torch.cuda.stream(stream):
            s, _ = binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                                   inp["kappa"], inp["mask"], saved=saved, stream=stream)
            g = binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                                 inp["kappa"], inp["mask"], inp["gs"], None, saved, scratch,
                                 stream=stream)
        return s, g

    ref = []
    for k in range(2):
        ref.append(run(k, torch.cuda.current_stream()))
        torch.cuda.synchronize()
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    for st in streams:
        st.wait_stream(torch.cuda.current_stream())
    got = [run(k, streams[k]) for k in range(2)]
    torch.cuda.synchronize()
    for (s0, g0), (s1, g1) in zip(ref, got):
        assert torch.equal(s0, s1)
        for key in g0:
            assert torch.equal(g0[key], g1[key]), key


def test_chained_layers_with_torch_kernels_between_calls():
    """The library's kernels start early behind the kernel before them in the stream and wait
    for it before reading: two layers chained through torch kernels (layer 1's spikes mixed
    into layer 2's input, layer 2's dL/dX reduced into layer 1's dL/dS), with no
    synchronisation between the calls, give the bits of the same chain run with a
    synchronisation after every operation."""
    w1 = workloads.Workload("ch1", T=8, B=3, N=2 * 128, K=8, G=1, C=2, inner=128, dtype="bf16",
                            psi="mh", reset="soft", seed=71)
    w2 = workloads.Workload("ch2", T=8, B=3, N=2 * 128, K=4, G=1, C=2, inner=128, dtype="bf16",
                            psi="mh", reset="hard", seed=72)
    c1, c2 = binding.config_of(w1), binding.config_of(w2)
    i1, i2 = (to_dev(workloads.make_inputs(w, "cpu")) for w in (w1, w2))
    p1 = [i1[k] for k in ("alpha", "xi", "zeta", "kappa")]
    p2 = [i2[k] for k in ("alpha", "xi", "zeta", "kappa")]
    mix = torch.randn(w2.K, generator=torch.Generator().manual_seed(5)).to("cuda", torch.bfloat16)

    def chain(sync):
        step = torch.cuda.synchronize if sync else (lambda: None)
        sv1, sc1 = binding.workspace(c1)
        sv2, sc2 = binding.workspace(c2)
        s1, _ = binding.forward(c1, i1["x"], *p1, None, saved=sv1)
        step()
        x2 = (s1.unsqueeze(-1) * mix + i2["x"]).contiguous()        # torch kernels
        step()
        s2, _ = binding.forward(c2, x2, *p2, None, saved=sv2)
        step()
        g2 = binding.backward(c2, x2, *p2, None, i2["gs"] * s2, None, sv2, sc2)
        step()
        gs1 = (g2["gx"].float() @ mix.float()).to(torch.bfloat16)     # torch kernels
        step()
        g1 = binding.backward(c1, i1["x"], *p1, None, gs1, None, sv1, sc1, want_beta=True)
        torch.cuda.synchronize()
        return [s1, s2] + [g2[k] for k in sorted(g2)] + [g1[k] for k in sorted(g1)]

    ref = chain(True)
    for _ in range(3):
        got = chain(False)
        for a, b in zip(ref, got):
            assert torch.equal(a, b)
