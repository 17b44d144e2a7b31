"""The C ABI driven from plain C99 (tests/c_host/dendsn_c_host.c), no Python in between.

* CPU: the program compiles as C99 against include/dendsn.h and links against libdendsn.so
  and the CUDA runtime (the header needs no C++ and no torch).
* GPU: it runs a seeded layer (T = 9: checkpoints; ragged chunks) and its outputs equal
  the Python binding's bit for bit, and the oracle within the parity tolerances.
"""
import os
import subprocess

import numpy as np
import pytest
import torch

import oracle
from paper_2412_06355_gb300 import binding, build, workloads

from parity import G_ATOL_REL, G_RTOL, V_ATOL, V_RTOL, assert_close, first_ambiguous_step

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "c_host", "dendsn_c_host.c")
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def compile_host(out_dir: str) -> str:
    lib = build.build()
    exe = os.path.join(out_dir, "dendsn_c_host")
    libdir = os.path.dirname(lib)
    cmd = ["gcc", "-std=c99", "-O2", "-Wall", "-Werror", "-I", build.INCLUDE,
           "-I", os.path.join(CUDA, "include"), SRC, "-o", exe,
           lib, f"-Wl,-rpath,{libdir}", "-L", os.path.join(CUDA, "lib64"), "-lcudart"]
    subprocess.run(cmd, check=True, capture_output=True, text=True)
    return exe


def test_c_host_compiles_and_links(tmp_path):
    exe = compile_host(str(tmp_path))
    assert os.path.exists(exe)


@pytest.mark.gpu
def test_c_host_runs_the_layer(tmp_path):
    if not torch.cuda.is_available():
        pytest.fail("needs a CUDA device")
    w = workloads.Workload("c_host", T=9, B=3, N=4 * 96, K=4, G=2, C=4, inner=96, dtype="f32",
                           psi="mh", reset="hard", seed=31)
    inp = workloads.make_inputs(w, "cpu")
    s_o, v_o = oracle.forward_layer(w, inp)
    amb = torch.from_numpy(first_ambiguous_step(v_o, w.theta) < w.T)
    gs = inp["gs"].clone()
    gs[:, amb] = 0
    d = str(tmp_path)
    with open(os.path.join(d, "cfg.txt"), "w") as f:
        f.write(f"{w.T} {w.B} {w.N} {w.K} {w.G} {w.C} {w.inner} 1 0\n")
    for name, t in (("x", inp["x"]), ("alpha", inp["alpha"]), ("xi", inp["xi"]),
                    ("zeta", inp["zeta"]), ("kappa", inp["kappa"]), ("gs", gs)):
        t.contiguous().numpy().astype(np.float32).tofile(os.path.join(d, f"{name}.bin"))
    exe = compile_host(d)
    r = subprocess.run([exe, d], capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    rd = lambda n, shape: np.fromfile(os.path.join(d, f"{n}.bin"), np.float32).reshape(shape)
    c = {"s": rd("spikes", (w.T, w.B, w.N)), "v": rd("v", (w.T, w.B, w.N)),
         "gx": rd("gx", (w.T, w.B, w.N, w.K)), "galpha": rd("galpha", (w.C, w.K)),
         "gxi": rd("gxi", (w.C, w.K)), "gzeta": rd("gzeta", (w.C, w.Kb)),
         "gkappa": rd("gkappa", (w.C, w.Kb))}
    # the same kernels through the Python binding: bit-identical
    cfg = binding.config_of(w)
    dev = {k: (None if v is None else v.cuda()) for k, v in inp.items()}
    saved, scratch = binding.workspace(cfg)
    s, v = binding.forward(cfg, dev["x"], dev["alpha"], dev["xi"], dev["zeta"], dev["kappa"],
                           None, want_v=True, saved=saved)
    g = binding.backward(cfg, dev["x"], dev["alpha"], dev["xi"], dev["zeta"], dev["kappa"],
                         None, gs.cuda(), None, saved, scratch)
    torch.cuda.synchronize()
    assert np.array_equal(c["s"], s.cpu().numpy()) and np.array_equal(c["v"], v.cpu().numpy())
    for k in ("gx", "galpha", "gxi", "gzeta", "gkappa"):
        assert np.array_equal(c[k], g[k].cpu().numpy()), k
    # and the oracle
    first = first_ambiguous_step(v_o, w.theta)
    t_idx = np.arange(w.T)[:, None, None]
    assert_close("V^s", c["v"], v_o, V_RTOL, 0.0, mask=t_idx <= first[None], atol_abs=V_ATOL)
    ref = oracle.backward_layer(w, inp, gs=gs)
    assert_close("grad_x", c["gx"], ref["gx"], G_RTOL, G_ATOL_REL)
    for k in ("galpha", "gxi", "gzeta", "gkappa"):
        assert_close(k, c[k], ref[k], G_RTOL, G_ATOL_REL)
