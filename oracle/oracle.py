"""ctypes wrapper of the C float64 oracle (dendsn_oracle.c).

TEST INFRASTRUCTURE ONLY: imported by the tests, the smoke check and the
benchmark's CPU-baseline leg, never by the product path.

Inputs are taken exactly as stored (float32, or bfloat16 widened exactly) and
converted to float64 before the C code sees them; all arithmetic is float64.
Parity status: pinned (closed forms, finite differences, an autograd
restatement and invariants; see tests/test_oracle_pins.py).
"""
from __future__ import annotations

import contextlib
import ctypes
import dataclasses
import os
import subprocess
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "dendsn_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lib = None


class _Cfg(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int32), ("M", ctypes.c_int32), ("K", ctypes.c_int32),
                ("G", ctypes.c_int32), ("C", ctypes.c_int32), ("psi", ctypes.c_int32),
                ("reset", ctypes.c_int32), ("stateless", ctypes.c_int32),
                ("residual", ctypes.c_int32), ("detach_reset", ctypes.c_int32),
                ("smooth_spike", ctypes.c_int32), ("theta", ctypes.c_double),
                ("beta", ctypes.c_double)]


@dataclasses.dataclass
class OracleConfig:
    T: int
    K: int
    G: int
    C: int
    psi: str = "mh"           # "mh" | "identity"
    reset: str = "hard"       # "hard" | "soft"
    theta: float = 1.0
    beta: float = 0.5
    stateless: bool = False
    residual: bool = False
    detach_reset: bool = False
    smooth_spike: bool = False

    @property
    def Kb(self) -> int:
        return self.K // self.G


def build(force: bool = False) -> str:
    """Compile the oracle with gcc into oracle/_build/liboracle.so."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or \
            os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-ffp-contract=off", "-shared",
                               "-fPIC", _SRC, "-o", tmp, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _configure(lib):
    P = ctypes.c_void_p
    for name, nargs in (("oracle_forward", 11), ("oracle_backward", 18),
                        ("oracle_lif_forward", 4), ("oracle_lif_backward", 5)):
        fn = getattr(lib, name)
        fn.restype = ctypes.c_int
        fn.argtypes = [ctypes.POINTER(_Cfg)] + [P] * (nargs - 1)
    return lib


def _load():
    global _lib
    if _lib is None:
        _lib = _configure(ctypes.CDLL(build()))
    return _lib


@contextlib.contextmanager
def using_library(path: str):
    """Test hook: run this wrapper against another build of the oracle (a mutant)."""
    global _lib
    saved = _lib
    _lib = _configure(ctypes.CDLL(path))
    try:
        yield
    finally:
        _lib = saved


def source_path() -> str:
    return _SRC


def to_f64(a) -> np.ndarray:
    """Exact widening of a stored float32 / bfloat16 tensor (torch or numpy)."""
    try:
        import torch
        if isinstance(a, torch.Tensor):
            a = a.detach().cpu()
            if a.dtype == torch.bfloat16:
                a = a.float()
            return np.ascontiguousarray(a.numpy().astype(np.float64))
    except ImportError:  # pragma: no cover
        pass
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _cfg(c: OracleConfig, M: int) -> _Cfg:
    return _Cfg(c.T, M, c.K, c.G, c.C, 1 if c.psi == "mh" else 0,
                0 if c.reset == "hard" else 1, int(c.stateless), int(c.residual),
                int(c.detach_reset), int(c.smooth_spike), float(c.theta), float(c.beta))


def _prep(c: OracleConfig, x, chan, mrow, alpha, xi, zeta, kappa, mask):
    x = to_f64(x)
    T, M, K = x.shape
    assert T == c.T and K == c.K, (x.shape, c)
    chan = np.ascontiguousarray(np.asarray(chan, dtype=np.int32))
    assert chan.shape == (M,) and (chan >= 0).all() and (chan < c.C).all()
    if mrow is not None:
        mrow = np.ascontiguousarray(np.asarray(mrow, dtype=np.int32))
        assert mrow.shape == (M,)
    p = [to_f64(alpha).reshape(c.C, c.K), to_f64(xi).reshape(c.C, c.K),
         to_f64(zeta).reshape(c.C, c.Kb), to_f64(kappa).reshape(c.C, c.Kb)]
    if mask is not None:
        try:
            import torch
            if isinstance(mask, torch.Tensor):
                mask = mask.cpu().numpy()
        except ImportError:  # pragma: no cover
            pass
        mask = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8))
        assert mask.ndim == 2 and mask.shape[1] == c.Kb
        if mrow is not None:
            assert (mrow < mask.shape[0]).all()
    return x, M, chan, mrow, p, mask


def forward(c: OracleConfig, x, chan, mrow, alpha, xi, zeta, kappa, mask=None):
    """Forward of M neurons. x: [T, M, K]. Returns (S, V), each [T, M] float64."""
    x, M, chan, mrow, p, mask = _prep(c, x, chan, mrow, alpha, xi, zeta, kappa, mask)
    s = np.zeros((c.T, M), np.float64)
    v = np.zeros((c.T, M), np.float64)
    cfg = _cfg(c, M)
    rc = _load().oracle_forward(ctypes.byref(cfg), _ptr(x), _ptr(chan), _ptr(mrow),
                                *[_ptr(a) for a in p], _ptr(mask), _ptr(s), _ptr(v))
    if rc != 0:
        raise RuntimeError("oracle_forward failed")
    return s, v


def backward(c: OracleConfig, x, chan, mrow, alpha, xi, zeta, kappa, mask, gs, gv=None,
             want_dvs: bool = False):
    """Backward of M neurons. Returns dict gx [T,M,K], galpha, gxi [C,K], gzeta, gkappa [C,Kb],
    gbeta [C] (dL/dbeta per channel; a layer-wide beta's gradient is the sum), and with
    want_dvs also dvs [T,M] = dL/dV^s[t]."""
    x, M, chan, mrow, p, mask = _prep(c, x, chan, mrow, alpha, xi, zeta, kappa, mask)
    gs = to_f64(gs).reshape(c.T, M)
    gv = None if gv is None else to_f64(gv).reshape(c.T, M)
    out = dict(gx=np.zeros((c.T, M, c.K)), galpha=np.zeros((c.C, c.K)),
               gxi=np.zeros((c.C, c.K)), gzeta=np.zeros((c.C, c.Kb)),
               gkappa=np.zeros((c.C, c.Kb)), gbeta=np.zeros(c.C))
    if want_dvs:
        out["dvs"] = np.zeros((c.T, M))
    cfg = _cfg(c, M)
    rc = _load().oracle_backward(ctypes.byref(cfg), _ptr(x), _ptr(chan), _ptr(mrow),
                                 *[_ptr(a) for a in p], _ptr(mask), _ptr(gs), _ptr(gv),
                                 _ptr(out["gx"]), _ptr(out["galpha"]), _ptr(out["gxi"]),
                                 _ptr(out["gzeta"]), _ptr(out["gkappa"]), _ptr(out["gbeta"]),
                                 _ptr(out.get("dvs")))
    if rc != 0:
        raise RuntimeError("oracle_backward failed")
    return out


@dataclasses.dataclass
class LIFConfig:
    """Point-neuron LIF layer (the DendSN soma driven directly by one current per neuron)."""
    T: int
    reset: str = "hard"
    theta: float = 1.0
    beta: float = 0.5
    detach_reset: bool = False
    smooth_spike: bool = False


def _lif_cfg(c: LIFConfig, M: int) -> _Cfg:
    return _Cfg(c.T, M, 1, 1, 1, 0, 0 if c.reset == "hard" else 1, 0, 0,
                int(c.detach_reset), int(c.smooth_spike), float(c.theta), float(c.beta))


def lif_forward(c: LIFConfig, x):
    """LIF forward of M neurons. x: [T, M] (or [T, ...]). Returns (S, V) float64, x's shape."""
    x = to_f64(x)
    shape = x.shape
    assert shape[0] == c.T, (shape, c)
    x = np.ascontiguousarray(x.reshape(c.T, -1))
    M = x.shape[1]
    s = np.zeros((c.T, M))
    v = np.zeros((c.T, M))
    cfg = _lif_cfg(c, M)
    if _load().oracle_lif_forward(ctypes.byref(cfg), _ptr(x), _ptr(s), _ptr(v)) != 0:
        raise RuntimeError("oracle_lif_forward failed")
    return s.reshape(shape), v.reshape(shape)


def lif_backward(c: LIFConfig, x, gs, gv=None):
    """LIF backward of M neurons; returns dL/dX with x's shape."""
    x = to_f64(x)
    shape = x.shape
    x = np.ascontiguousarray(x.reshape(c.T, -1))
    M = x.shape[1]
    gs = np.ascontiguousarray(to_f64(gs).reshape(c.T, M))
    gv = None if gv is None else np.ascontiguousarray(to_f64(gv).reshape(c.T, M))
    gx = np.zeros((c.T, M))
    cfg = _lif_cfg(c, M)
    if _load().oracle_lif_backward(ctypes.byref(cfg), _ptr(x), _ptr(gs), _ptr(gv), _ptr(gx)) != 0:
        raise RuntimeError("oracle_lif_backward failed")
    return gx.reshape(shape)


def layer_channels(B: int, N: int, C: int, inner: int, mask_per_neuron: bool):
    """Channel and mask row of every neuron of a [B, N] layer, flattened b-major.

    Neurons at the spatial positions of one channel share parameters (Methods,
    "Dendritic spiking neural networks", constraint 3): c(n) = (n // inner) % C.
    The mask is indexed by channel (Eq. methods-dbg-mask, [C, B] shape) or, when
    mask_per_neuron, by the neuron index n within a sample.
    """
    n = np.arange(N, dtype=np.int64)
    chan = ((n // inner) % C).astype(np.int32)
    chan = np.tile(chan, B)
    mrow = np.tile(n.astype(np.int32), B) if mask_per_neuron else chan.copy()
    return chan, mrow


def _cfg_of(w, **over) -> OracleConfig:
    kw = dict(T=w.T, K=w.K, G=w.G, C=w.C, psi=w.psi, reset=w.reset, theta=w.theta,
              beta=w.beta, stateless=w.stateless, residual=w.residual,
              detach_reset=w.detach_reset)
    kw.update(over)
    return OracleConfig(**kw)


def layer_x(w, x) -> np.ndarray:
    """A layer's input currents as [T, B*N, K] float64, whatever layout they are stored in.

    "kinner": [T, B, N, K]. "paper": a conv layer's output channels grouped as
    (C_o, P, H, W) (Methods, "Dendritic spiking neural networks"), i.e.
    [T, B, N / inner, K, inner] with inner = H*W: compartment k of neuron n sits at
    [n // inner, k, n % inner].
    """
    x = to_f64(x)
    if getattr(w, "layout", "kinner") == "paper":
        x = x.reshape(w.T, w.B, w.N // w.inner, w.K, w.inner).transpose(0, 1, 2, 4, 3)
    return np.ascontiguousarray(x.reshape(w.T, w.B * w.N, w.K))


def layer_gx(w, gx: np.ndarray) -> np.ndarray:
    """[T, B*N, K] -> the layout layer_x reads (gradients share the input's layout)."""
    if getattr(w, "layout", "kinner") == "paper":
        gx = gx.reshape(w.T, w.B, w.N // w.inner, w.inner, w.K).transpose(0, 1, 2, 4, 3)
        return np.ascontiguousarray(gx)
    return gx.reshape(w.T, w.B, w.N, w.K)


def forward_layer(w, inp, **over):
    """Oracle forward of a whole workload `w` with inputs from make_inputs."""
    chan, mrow = layer_channels(w.B, w.N, w.C, w.inner, w.mask_per_neuron)
    x = layer_x(w, inp["x"])
    s, v = forward(_cfg_of(w, **over), x, chan, mrow, inp["alpha"], inp["xi"],
                   inp["zeta"], inp["kappa"], inp.get("mask"))
    return s.reshape(w.T, w.B, w.N), v.reshape(w.T, w.B, w.N)


def backward_layer(w, inp, gs=None, want_dvs=False, **over):
    """Oracle backward of a whole workload `w`; gs overrides inp['gs']."""
    chan, mrow = layer_channels(w.B, w.N, w.C, w.inner, w.mask_per_neuron)
    x = layer_x(w, inp["x"])
    gs = inp["gs"] if gs is None else gs
    out = backward(_cfg_of(w, **over), x, chan, mrow, inp["alpha"], inp["xi"], inp["zeta"],
                   inp["kappa"], inp.get("mask"), gs, inp.get("gv"), want_dvs=want_dvs)
    out["gx"] = layer_gx(w, out["gx"])
    if want_dvs:
        out["dvs"] = out["dvs"].reshape(w.T, w.B, w.N)
    return out
