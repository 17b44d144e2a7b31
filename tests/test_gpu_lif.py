"""GPU parity of the point-neuron LIF layer (the speed baseline) against its float64 oracle.

Same tolerances and ambiguous-step handling as the DendSN parity tests (tests/parity.py):
V within 1e-6 + 1e-5 |V|, spikes identical before the first step whose oracle potential
lies within 1e-5 of the threshold, gradients rtol 1e-4 (bf16 grad_x 2e-2), neurons with an
ambiguous step given zero upstream gradient on both sides.
Covers the vector (4 neurons per thread) and scalar kernels, 4- and 8-step chunks with
ragged tails and checkpoints, both resets, a detached reset, grad_v, bf16, empty layers
and the two full-size layers the benchmark times, on sampled neurons.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2412_06355_gb300 import binding, workloads

from parity import (BF16_ATOL_REL, BF16_RTOL, G_ATOL_REL, G_RTOL, V_ATOL, V_RTOL,
                    assert_close, first_ambiguous_step)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("these tests need a CUDA device")
    binding.load()
    oracle.build()


def run_lif(cfg, x, gs, gv):
    saved = binding.lif_workspace(cfg)
    s, v = binding.lif_forward(cfg, x, want_v=True, saved=saved)
    gx = binding.lif_backward(cfg, x, gs, gv, saved)
    # the production forward (no V output) gives the same spikes and checkpoints
    saved2 = binding.lif_workspace(cfg)
    s2, _ = binding.lif_forward(cfg, x, want_v=False, saved=saved2)
    torch.cuda.synchronize()
    assert torch.equal(s, s2)
    if saved is not None:
        used = ((cfg.T + 7) // 8 - 1) * cfg.B * cfg.N * 4      # the rest is alignment padding
        assert torch.equal(saved[:used], saved2[:used])
    return s, v, gx


def check_lif(T, B, N, dtype="f32", reset="hard", detach=False, theta=1.0, beta=0.5,
              with_gv=True, seed=0, offset=0):
    inp = workloads.make_lif_inputs(T, B, N + offset, dtype, seed, with_gv=with_gv)
    x = inp["x"][..., offset:]
    gs = inp["gs"][..., offset:].clone()
    gv = None if inp["gv"] is None else inp["gv"][..., offset:].clone()
    oc = oracle.LIFConfig(T=T, reset=reset, theta=theta, beta=beta, detach_reset=detach)
    s_o, v_o = oracle.lif_forward(oc, x)
    first = first_ambiguous_step(v_o, theta)
    amb = torch.from_numpy(first < T)
    gs[:, amb] = 0
    if gv is not None:
        gv[:, amb] = 0
    cfg = binding.make_lif_config(T, B, N, dtype, reset, theta, beta, detach)
    dev = lambda t: None if t is None else t.contiguous().cuda()
    xd = dev(x)
    if offset:
        # x starts `offset` elements into its buffer: not 16-byte aligned (scalar kernels)
        buf = torch.empty(T * B * N + offset, dtype=x.dtype, device="cuda")
        xd = buf[offset:].view(T, B, N)
        xd.copy_(x)
    s, v, gx = run_lif(cfg, xd, dev(gs), dev(gv))
    gx_o = oracle.lif_backward(oc, x, gs, gv)
    t_idx = np.arange(T)[:, None, None]
    assert_close("V", oracle.to_f64(v), v_o, V_RTOL, 0.0, mask=t_idx <= first[None],
                 atol_abs=V_ATOL)
    got_s = oracle.to_f64(s)
    sm = t_idx < first[None]
    assert np.array_equal(got_s[sm], s_o[sm])
    assert set(np.unique(got_s).tolist()) <= {0.0, 1.0}
    rt, ar = (BF16_RTOL, BF16_ATOL_REL) if dtype == "bf16" else (G_RTOL, G_ATOL_REL)
    assert_close("grad_x", oracle.to_f64(gx), gx_o, rt, ar)
    return float(s_o.mean())


@pytest.mark.parametrize("T", [1, 3, 4, 5, 8, 9, 16, 17, 64])
@pytest.mark.parametrize("N", [1000, 1001])
def test_lif_lengths_and_tails(T, N):
    assert check_lif(T, 3, N, seed=T) > 0.0


@pytest.mark.parametrize("kw", [dict(reset="soft"), dict(detach=True),
                                dict(reset="soft", detach=True), dict(with_gv=False),
                                dict(theta=0.5, beta=0.9), dict(beta=0.0),
                                dict(dtype="bf16"), dict(dtype="bf16", reset="soft", T=12)],
                         ids=lambda kw: "-".join(f"{k}={v}" for k, v in kw.items()))
def test_lif_variants(kw):
    args = dict(T=10, B=2, N=1024)
    args.update(kw)
    check_lif(**args)


def test_lif_misaligned_view_takes_the_scalar_kernel():
    check_lif(9, 2, 1024, offset=1)


def test_lif_empty():
    cfg = binding.make_lif_config(0, 2, 8)
    x = torch.empty(0, 2, 8, device="cuda")
    s, _ = binding.lif_forward(cfg, x)
    assert s.numel() == 0
    cfg = binding.make_lif_config(4, 0, 8)
    x = torch.empty(4, 0, 8, device="cuda")
    assert binding.lif_backward(cfg, x, x.clone()).numel() == 0


@pytest.mark.parametrize("N", [131072, 131072 * 4])
def test_lif_full_size_sampled(N):
    """The two LIF layers the benchmark times, compared on 3000 sampled neurons."""
    T, B = 4, 64
    inp = workloads.make_lif_inputs(T, B, N, "f32", seed=7, device="cuda")
    cfg = binding.make_lif_config(T, B, N)
    rng = np.random.default_rng(1)
    flat = np.sort(rng.choice(B * N, 3000, replace=False))
    bt, nt = torch.from_numpy(flat // N).cuda(), torch.from_numpy(flat % N).cuda()
    oc = oracle.LIFConfig(T=T)
    xs = inp["x"][:, bt, nt].cpu()
    s_o, v_o = oracle.lif_forward(oc, xs)
    first = first_ambiguous_step(v_o, 1.0)
    keep = torch.from_numpy(first == T).cuda()
    gs = torch.zeros_like(inp["gs"])
    gs[:, bt[keep], nt[keep]] = inp["gs"][:, bt[keep], nt[keep]]
    s, v = binding.lif_forward(cfg, inp["x"], want_v=True)
    gx = binding.lif_backward(cfg, inp["x"], gs)
    torch.cuda.synchronize()
    t_idx = np.arange(T)[:, None]
    assert_close("V", oracle.to_f64(v[:, bt, nt]), v_o, V_RTOL, 0.0,
                 mask=t_idx <= first[None], atol_abs=V_ATOL)
    sm = t_idx < first[None]
    assert np.array_equal(oracle.to_f64(s[:, bt, nt])[sm], s_o[sm])
    gx_o = oracle.lif_backward(oc, xs, gs[:, bt, nt].cpu())
    assert_close("grad_x", oracle.to_f64(gx[:, bt, nt]), gx_o, G_RTOL, G_ATOL_REL)
    gx[:, bt, nt] = 0
    assert torch.count_nonzero(gx).item() == 0
