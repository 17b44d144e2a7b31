"""The scratch-free backward (dendsn_backward_noalloc) against dendsn_backward.

Some callers cannot give the library a device scratch buffer (a C host that only holds
device pointers for the tensors, or a runtime that must not allocate per call); for them
the library keeps its own fixed buffer. These checks call both entry points through the
C ABI on the same inputs and require bit-identical gradients (both run the same kernels
in the same order, only the scratch address differs), on two calls in a row with
different layer sizes, so that what the first call leaves in the shared buffer cannot
leak into the second. This file sorts last so that a run that
stops at its first failure has already run every other test; it also passes on its own
in a fresh process (the first call on the device performs the one-time set-up).
"""
import ctypes

import pytest
import torch

from paper_2412_06355_gb300 import binding, workloads

from parity import to_dev

pytestmark = pytest.mark.gpu

CASES = [
    # large first (a transformer-token layer: per-neuron mask, many channels) ...
    workloads.scaled(workloads.WORKLOADS["token_dbg"], B=4),
    # ... then a smaller conv-shaped layer with checkpoints and bf16 inputs
    workloads.Workload("small", T=12, B=3, N=2 * 256, K=8, G=1, C=2, inner=256, dtype="bf16",
                       psi="mh", reset="soft", seed=77),
]


def run_both(w):
    cfg = binding.config_of(w)
    inp = to_dev(workloads.make_inputs(w, "cpu", with_gv=True))
    saved, scratch = binding.workspace(cfg)
    binding.forward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"],
                    inp["mask"], saved=saved)
    ref = binding.backward(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"], inp["kappa"],
                           inp["mask"], inp["gs"], inp["gv"], saved, scratch)
    C, K, Kb = cfg.C, cfg.K, cfg.K // cfg.G
    got = dict(gx=torch.full_like(inp["x"], float("nan")),
               galpha=torch.full((C, K), float("nan"), device="cuda"),
               gxi=torch.full((C, K), float("nan"), device="cuda"),
               gzeta=torch.full((C, Kb), float("nan"), device="cuda"),
               gkappa=torch.full((C, Kb), float("nan"), device="cuda"))
    binding.dendsn_backward_noalloc(cfg, inp["x"], inp["alpha"], inp["xi"], inp["zeta"],
                                    inp["kappa"], inp["mask"], inp["gs"], inp["gv"], saved,
                                    got["gx"], got["galpha"], got["gxi"], got["gzeta"],
                                    got["gkappa"])
    torch.cuda.synchronize()
    return ref, got


def test_noalloc_backward_matches_backward_twice_in_a_row():
    if not torch.cuda.is_available():
        pytest.fail("needs a CUDA device")
    for w in CASES:
        ref, got = run_both(w)
        for k in ("gx", "galpha", "gxi", "gzeta", "gkappa"):
            assert torch.equal(got[k], ref[k]), f"{w.name} {k} differs from dendsn_backward"


def test_noalloc_rejects_layers_beyond_its_buffer():
    if not torch.cuda.is_available():
        pytest.fail("needs a CUDA device")
    # 65536 channels of one neuron each with 16 compartments: every block keeps
    # partials for all the channels of its columns, 16 MiB in all, twice the built-in 8 MiB
    w = workloads.Workload("huge", T=1, B=32, N=65536, K=16, G=1, C=65536, inner=1,
                           dtype="f32", psi="mh", reset="hard")
    cfg = binding.config_of(w)
    _, need = binding.dendsn_workspace_size(cfg)
    assert need > 8 << 20
    # the library itself must refuse before touching any tensor, so it is called
    # directly (the Python wrapper would already refuse these 64-byte tensors)
    d = torch.empty(16, device="cuda")
    lib = binding.load()
    fn = lib.dendsn_backward_noalloc
    fn.argtypes = [ctypes.POINTER(binding.dendsn_config)] + [ctypes.c_void_p] * 15
    fn.restype = ctypes.c_int
    p = d.data_ptr()
    st = fn(ctypes.byref(cfg), p, p, p, p, p, None, p, None, None, p, p, p, p, p, None)
    msg = lib.dendsn_last_error().decode()
    assert st == 2 and "8388608" in msg and str(need) in msg, (st, msg)
