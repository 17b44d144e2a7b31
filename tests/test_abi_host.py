"""Host-side checks of the C ABI: no GPU needed, no kernel is launched.

* libdendsn.so builds for sm_103a and loads;
* it exports every function include/dendsn.h declares;
* the Python mirror of dendsn_config has the C layout (checked with gcc);
* argument validation returns the documented status before any launch;
* workspace sizes follow the checkpoint layout.
"""
import ctypes
import os
import re
import subprocess
import tempfile

import pytest

from paper_2412_06355_gb300 import binding
from paper_2412_06355_gb300.binding import make_config

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dendsn.h")


@pytest.fixture(scope="module")
def lib():
    return binding.load()


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(dendsn_\w+)\s*\(", src, re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("dendsn_forward", "dendsn_backward", "dendsn_workspace_size",
                     "dendsn_status_string", "dendsn_last_error"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    out = subprocess.run(["nm", "-D", "--defined-only", binding.library_path()],
                         capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\s[TW]\s+(\w+)$", out, re.M))
    for name in declared_functions():
        assert name in exported, name
        assert hasattr(lib, name)


@pytest.mark.parametrize("struct", [binding.dendsn_config, binding.dendsn_lif_config],
                         ids=lambda s: s.__name__)
def test_config_layout_matches_c(struct):
    name = struct.__name__
    fields = [f[0] for f in struct._fields_]
    prog = "#include <stdio.h>\n#include <stddef.h>\n#include \"dendsn.h\"\nint main(void){\n"
    prog += f'printf("%zu\\n", sizeof({name}));\n'
    for f in fields:
        prog += f'printf("%zu\\n", offsetof({name}, {f}));\n'
    prog += "return 0;}\n"
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        open(c, "w").write(prog)
        subprocess.check_call(["gcc", "-std=c99", "-I", os.path.join(ROOT, "include"), c, "-o", exe])
        vals = [int(v) for v in subprocess.check_output([exe]).split()]
    assert vals[0] == ctypes.sizeof(struct)
    for f, off in zip(fields, vals[1:]):
        assert getattr(struct, f).offset == off, f


def status_of(fn, *args):
    try:
        fn(*args)
    except binding.DendSNError as e:
        return e.status
    return 0


@pytest.mark.parametrize("kw,status", [
    (dict(K=3), 2),                       # valid, but K=3 is not compiled in
    (dict(K=4, G=3), 1),                  # G does not divide K
    (dict(K=32), 2),                      # K not compiled in
    (dict(K=8, G=8), 2),                  # G larger than the per-lane share
    (dict(N=100, C=3, inner=10), 1),      # N not a multiple of C*inner
    (dict(T=-1), 1),
    (dict(C=0), 1),
    (dict(surrogate=1), 2),               # only the arctan surrogate
])
def test_workspace_size_validation(kw, status):
    base = dict(T=4, B=2, N=64, K=4, G=1, C=4, inner=16)
    base.update(kw)
    surrogate = base.pop("surrogate", 0)
    cfg = make_config(**base, surrogate=surrogate)
    assert status_of(binding.dendsn_workspace_size, cfg) == status


def test_bad_flag_values_rejected():
    cfg = make_config(T=4, B=2, N=64, K=4, C=4, inner=16)
    cfg.psi = 7
    assert status_of(binding.dendsn_workspace_size, cfg) == 1
    cfg.psi = 1
    cfg.reset = 2
    assert status_of(binding.dendsn_workspace_size, cfg) == 1
    cfg.reset = 0
    cfg.theta = float("nan")
    assert status_of(binding.dendsn_workspace_size, cfg) == 1


def test_workspace_sizes_follow_checkpoint_layout():
    # T <= 8 is recomputed from x alone: no saved state
    for T in (1, 4, 5, 8):
        saved, scratch = binding.dendsn_workspace_size(make_config(T=T, B=2, N=256, K=4, C=2, inner=128))
        assert saved == 0 and scratch > 0
    # bfloat16 rows of one chunk of whole 8-compartment neurons (the phased backward): the
    # forward keeps V^s, T x B x N float32
    B, N = 3, 256
    for T, dt in ((8, "bf16"), (4, "bf16")):
        saved, _ = binding.dendsn_workspace_size(make_config(T=T, B=B, N=N, K=8, C=2, inner=128,
                                                             dtype=dt))
        assert saved == T * B * N * 4, (T, dt)
    # not those layers: float32 (T = 8 phased without a kept V^s; T = 4 split lanes), T
    # between chunk lengths, the residual term, the paper layout, two compartments per branch
    for kw in (dict(T=8), dict(T=4), dict(T=6, dtype="bf16"), dict(T=8, dtype="bf16", residual=True),
               dict(T=8, dtype="bf16", layout="paper"), dict(T=8, dtype="bf16", G=2)):
        saved, _ = binding.dendsn_workspace_size(make_config(**dict(dict(B=B, N=N, K=8, C=2,
                                                                         inner=128), **kw)))
        assert saved == 0, kw
    # T = 64, chunk 8: 7 checkpoints of (K V^d + 1 V^s) float32 per neuron
    B, N, K = 2, 256, 4
    saved, _ = binding.dendsn_workspace_size(make_config(T=64, B=B, N=N, K=K, C=2, inner=128))
    assert saved == 7 * B * N * (K + 1) * 4
    saved, _ = binding.dendsn_workspace_size(make_config(T=17, B=B, N=N, K=K, C=2, inner=128))
    assert saved == 2 * B * N * (K + 1) * 4


def test_null_and_misaligned_pointers_rejected_before_launch(lib):
    cfg = make_config(T=4, B=1, N=64, K=4, C=4, inner=16)
    P = ctypes.c_void_p
    ok = P(4096)          # never dereferenced: validation fails first
    st = lib.dendsn_forward(ctypes.byref(cfg), None, ok, ok, ok, ok, None, ok, None, None, None)
    assert st == 1 and b"NULL" in lib.dendsn_last_error()
    st = lib.dendsn_forward(ctypes.byref(cfg), P(4100), ok, ok, ok, ok, None, ok, None, None, None)
    assert st == 3
    st = lib.dendsn_backward(ctypes.byref(cfg), ok, ok, ok, ok, ok, None, ok, None, None, ok,
                             ok, ok, ok, ok, None, None)
    assert st == 1          # scratch is NULL
    cfg64 = make_config(T=64, B=1, N=64, K=4, C=4, inner=16)
    st = lib.dendsn_backward(ctypes.byref(cfg64), ok, ok, ok, ok, ok, None, ok, None, None, ok,
                             ok, ok, ok, ok, ok, None)
    assert st == 1 and b"checkpoints" in lib.dendsn_last_error()


def test_layout_flag_validated():
    cfg = make_config(T=4, B=2, N=64, K=4, C=4, inner=16, layout="paper")
    assert cfg.layout == binding.LAYOUT_PAPER
    assert status_of(binding.dendsn_workspace_size, cfg) == 0
    cfg.layout = 2
    assert status_of(binding.dendsn_workspace_size, cfg) == 1


def test_binding_refuses_undersized_tensors(lib):
    """Sizes are checked on the host before any pointer reaches the library."""
    import torch
    cfg = make_config(T=4, B=2, N=64, K=4, C=4, inner=16, layout="paper")
    x = torch.zeros(4, 2, 4, 4, 16)                       # the paper layout: right size
    p = [torch.zeros(4, 4) for _ in range(4)]
    with pytest.raises(ValueError, match="spikes"):
        binding.dendsn_forward(cfg, x, *p, None, torch.zeros(4, 2, 4))   # [T, B, N/inner]
    with pytest.raises(ValueError, match="x:"):
        binding.dendsn_forward(cfg, x[:, :1], *p, None, torch.zeros(4, 2, 64))
    with pytest.raises(ValueError, match="scratch"):
        binding.dendsn_backward(cfg, x, *p, None, torch.zeros(4, 2, 64), None, None,
                                torch.zeros_like(x), *p, torch.zeros(1))


def test_lif_validation_and_workspace(lib):
    mk = binding.make_lif_config
    assert binding.dendsn_lif_workspace_size(mk(T=8, B=2, N=10)) == 0
    assert binding.dendsn_lif_workspace_size(mk(T=9, B=2, N=10)) == 80      # 1 x 20 x 4 B
    assert binding.dendsn_lif_workspace_size(mk(T=64, B=3, N=7)) == (7 * 21 * 4 + 15) // 16 * 16
    for bad in (dict(T=-1), dict(reset=2), dict(x_dtype=5), dict(theta=float("inf"))):
        cfg = mk(T=4, B=2, N=10)
        for k, v in bad.items():
            setattr(cfg, k, v)
        assert status_of(binding.dendsn_lif_workspace_size, cfg) == 1, bad
    P = ctypes.c_void_p
    cfg = mk(T=4, B=1, N=64)
    assert lib.dendsn_lif_forward(ctypes.byref(cfg), None, P(4096), None, None, None) == 1
    assert lib.dendsn_lif_forward(ctypes.byref(cfg), P(4098), P(4096), None, None, None) == 3
    cfg = mk(T=20, B=1, N=64)       # needs checkpoints
    assert lib.dendsn_lif_backward(ctypes.byref(cfg), P(4096), P(4096), None, None, P(4096),
                                   None) == 1


def test_status_strings(lib):
    for code in range(5):
        assert lib.dendsn_status_string(code)
