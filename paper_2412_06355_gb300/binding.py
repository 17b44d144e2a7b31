"""Thin ctypes binding of libdendsn (include/dendsn.h).

Argument marshalling only: every step of the DendSN forward and backward runs in
the library's CUDA kernels. torch supplies device memory and the current stream.
There is no fallback: if the library cannot be loaded, every call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional

import torch

from . import build as _build

F32, BF16 = 0, 1
PSI_IDENTITY, PSI_MEXHAT = 0, 1
RESET_HARD, RESET_SOFT = 0, 1
SG_ATAN = 0

STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported configuration",
          3: "misaligned pointer", 4: "CUDA error"}


class DendSNError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str):
        super().__init__(f"{fn}: {STATUS.get(status, status)}: {msg}")
        self.status = status


class dendsn_config(ctypes.Structure):
    """Mirror of the C struct dendsn_config."""
    _fields_ = [("T", ctypes.c_int32), ("B", ctypes.c_int32), ("N", ctypes.c_int32),
                ("K", ctypes.c_int32), ("G", ctypes.c_int32), ("C", ctypes.c_int32),
                ("inner", ctypes.c_int32), ("x_dtype", ctypes.c_int32),
                ("psi", ctypes.c_int32), ("reset", ctypes.c_int32),
                ("surrogate", ctypes.c_int32), ("theta", ctypes.c_float),
                ("beta", ctypes.c_float), ("detach_reset", ctypes.c_int32),
                ("mask_per_neuron", ctypes.c_int32), ("stateless", ctypes.c_int32),
                ("residual", ctypes.c_int32), ("layout", ctypes.c_int32)]

    @property
    def Kb(self) -> int:
        return self.K // self.G


LAYOUT_KINNER, LAYOUT_PAPER = 0, 1


def make_config(T, B, N, K, G=1, C=1, inner=1, dtype="f32", psi="mh", reset="hard",
                theta=1.0, beta=0.5, detach_reset=False, mask_per_neuron=False,
                stateless=False, residual=False, surrogate=SG_ATAN,
                layout="kinner") -> dendsn_config:
    return dendsn_config(T, B, N, K, G, C, inner, BF16 if dtype == "bf16" else F32,
                         PSI_MEXHAT if psi == "mh" else PSI_IDENTITY,
                         RESET_SOFT if reset == "soft" else RESET_HARD, surrogate,
                         float(theta), float(beta), int(detach_reset), int(mask_per_neuron),
                         int(stateless), int(residual),
                         LAYOUT_PAPER if layout == "paper" else LAYOUT_KINNER)


def config_of(w) -> dendsn_config:
    """Config of a workloads.Workload."""
    return make_config(w.T, w.B, w.N, w.K, w.G, w.C, w.inner, w.dtype, w.psi, w.reset,
                       w.theta, w.beta, w.detach_reset, w.mask_per_neuron, w.stateless,
                       w.residual, layout=w.layout)


class dendsn_lif_config(ctypes.Structure):
    """Mirror of the C struct dendsn_lif_config (the point-neuron LIF layer)."""
    _fields_ = [("T", ctypes.c_int32), ("B", ctypes.c_int32), ("N", ctypes.c_int32),
                ("x_dtype", ctypes.c_int32), ("reset", ctypes.c_int32),
                ("theta", ctypes.c_float), ("beta", ctypes.c_float),
                ("detach_reset", ctypes.c_int32)]


def make_lif_config(T, B, N, dtype="f32", reset="hard", theta=1.0, beta=0.5,
                    detach_reset=False) -> dendsn_lif_config:
    return dendsn_lif_config(T, B, N, BF16 if dtype == "bf16" else F32,
                             RESET_SOFT if reset == "soft" else RESET_HARD, float(theta),
                             float(beta), int(detach_reset))


_lib = None
_lock = threading.Lock()


def library_path() -> str:
    return _build.LIB


def load() -> ctypes.CDLL:
    """Load libdendsn.so, building it first when it is missing or stale."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            lib = ctypes.CDLL(path)
            P, cfgp = ctypes.c_void_p, ctypes.POINTER(dendsn_config)
            lib.dendsn_workspace_size.argtypes = [cfgp, ctypes.POINTER(ctypes.c_size_t),
                                                  ctypes.POINTER(ctypes.c_size_t)]
            lib.dendsn_forward.argtypes = [cfgp] + [P] * 10
            lib.dendsn_backward.argtypes = [cfgp] + [P] * 16
            lib.dendsn_backward_plif.argtypes = [cfgp] + [P] * 17
            lib.dendsn_backward_plif.restype = ctypes.c_int
            lcfgp = ctypes.POINTER(dendsn_lif_config)
            lib.dendsn_lif_workspace_size.argtypes = [lcfgp, ctypes.POINTER(ctypes.c_size_t)]
            lib.dendsn_lif_forward.argtypes = [lcfgp] + [P] * 5
            lib.dendsn_lif_backward.argtypes = [lcfgp] + [P] * 6
            for fn in (lib.dendsn_workspace_size, lib.dendsn_forward, lib.dendsn_backward,
                       lib.dendsn_lif_workspace_size, lib.dendsn_lif_forward,
                       lib.dendsn_lif_backward):
                fn.restype = ctypes.c_int
            lib.dendsn_status_string.argtypes = [ctypes.c_int]
            lib.dendsn_status_string.restype = ctypes.c_char_p
            lib.dendsn_last_error.argtypes = []
            lib.dendsn_last_error.restype = ctypes.c_char_p
            lib.dendsn_launch_count.argtypes = []
            lib.dendsn_launch_count.restype = ctypes.c_uint64
            _lib = lib
    return _lib


def _check(fn: str, status: int):
    if status != 0:
        raise DendSNError(fn, status, load().dendsn_last_error().decode())


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("DendSN tensors must live on a CUDA device")
    if not t.is_contiguous():
        raise ValueError("DendSN tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def launch_count() -> int:
    """Kernels the library has enqueued since it was loaded."""
    return int(load().dendsn_launch_count())


def dendsn_workspace_size(cfg: dendsn_config):
    """(saved_bytes, scratch_bytes) for this config."""
    s, w = ctypes.c_size_t(0), ctypes.c_size_t(0)
    _check("dendsn_workspace_size",
           load().dendsn_workspace_size(ctypes.byref(cfg), ctypes.byref(s), ctypes.byref(w)))
    return int(s.value), int(w.value)


def _need(cfg, **tensors):
    """Refuses on the host any tensor smaller than what the config makes the kernels touch."""
    T, B, N, K, C, Kb = cfg.T, cfg.B, cfg.N, cfg.K, cfg.C, cfg.K // cfg.G
    sx = 2 if cfg.x_dtype == BF16 else 4
    elems = {"x": T * B * N * K * sx, "grad_x": T * B * N * K * sx,
             "spikes": T * B * N * sx, "grad_spikes": T * B * N * sx,
             "v_out": T * B * N * 4, "grad_v": T * B * N * 4,
             "alpha": C * K * 4, "xi": C * K * 4, "grad_alpha": C * K * 4, "grad_xi": C * K * 4,
             "zeta": C * Kb * 4, "kappa": C * Kb * 4, "grad_zeta": C * Kb * 4,
             "grad_kappa": C * Kb * 4, "mask": (N if cfg.mask_per_neuron else C) * Kb,
             "grad_beta": C * 4}
    sizes = None
    for name, t in tensors.items():
        if t is None:
            continue
        if name in ("saved", "scratch"):
            if sizes is None:
                sizes = dict(zip(("saved", "scratch"), dendsn_workspace_size(cfg)))
            need = sizes[name]
        else:
            need = elems[name]
        have = t.numel() * t.element_size()
        if have < need:
            raise ValueError(f"{name}: {have} bytes, the config needs {need}")


def dendsn_forward(cfg, x, alpha, xi, zeta, kappa, mask, spikes, v_out=None, saved=None,
                   stream=None):
    _need(cfg, x=x, alpha=alpha, xi=xi, zeta=zeta, kappa=kappa, mask=mask, spikes=spikes,
          v_out=v_out, saved=saved)
    _check("dendsn_forward", load().dendsn_forward(
        ctypes.byref(cfg), _ptr(x), _ptr(alpha), _ptr(xi), _ptr(zeta), _ptr(kappa),
        _ptr(mask), _ptr(spikes), _ptr(v_out), _ptr(saved), _stream(stream)))


def dendsn_backward(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved, grad_x,
                    grad_alpha, grad_xi, grad_zeta, grad_kappa, scratch, stream=None):
    _need(cfg, x=x, alpha=alpha, xi=xi, zeta=zeta, kappa=kappa, mask=mask,
          grad_spikes=grad_spikes, grad_v=grad_v, saved=saved, grad_x=grad_x,
          grad_alpha=grad_alpha, grad_xi=grad_xi, grad_zeta=grad_zeta, grad_kappa=grad_kappa,
          scratch=scratch)
    _check("dendsn_backward", load().dendsn_backward(
        ctypes.byref(cfg), _ptr(x), _ptr(alpha), _ptr(xi), _ptr(zeta), _ptr(kappa),
        _ptr(mask), _ptr(grad_spikes), _ptr(grad_v), _ptr(saved), _ptr(grad_x),
        _ptr(grad_alpha), _ptr(grad_xi), _ptr(grad_zeta), _ptr(grad_kappa), _ptr(scratch),
        _stream(stream)))


def dendsn_backward_plif(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                         grad_x, grad_alpha, grad_xi, grad_zeta, grad_kappa, grad_beta, scratch,
                         stream=None):
    """dendsn_backward plus grad_beta [C], the gradient of a learnable somatic decay."""
    _need(cfg, x=x, alpha=alpha, xi=xi, zeta=zeta, kappa=kappa, mask=mask,
          grad_spikes=grad_spikes, grad_v=grad_v, saved=saved, grad_x=grad_x,
          grad_alpha=grad_alpha, grad_xi=grad_xi, grad_zeta=grad_zeta, grad_kappa=grad_kappa,
          grad_beta=grad_beta, scratch=scratch)
    _check("dendsn_backward_plif", load().dendsn_backward_plif(
        ctypes.byref(cfg), _ptr(x), _ptr(alpha), _ptr(xi), _ptr(zeta), _ptr(kappa),
        _ptr(mask), _ptr(grad_spikes), _ptr(grad_v), _ptr(saved), _ptr(grad_x),
        _ptr(grad_alpha), _ptr(grad_xi), _ptr(grad_zeta), _ptr(grad_kappa), _ptr(grad_beta),
        _ptr(scratch), _stream(stream)))


_noalloc_ready = False


def dendsn_backward_noalloc(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                            grad_x, grad_alpha, grad_xi, grad_zeta, grad_kappa, stream=None):
    """dendsn_backward without a scratch buffer (the library's built-in 8 MiB one).

    For callers that cannot allocate device scratch memory per call; see the header
    for the sharing rules of the built-in buffer.
    """
    global _noalloc_ready
    _need(cfg, x=x, alpha=alpha, xi=xi, zeta=zeta, kappa=kappa, mask=mask,
          grad_spikes=grad_spikes, grad_v=grad_v, saved=saved, grad_x=grad_x,
          grad_alpha=grad_alpha, grad_xi=grad_xi, grad_zeta=grad_zeta, grad_kappa=grad_kappa)
    lib = load()
    if not _noalloc_ready:
        lib.dendsn_backward_noalloc.argtypes = [ctypes.POINTER(dendsn_config)] + \
            [ctypes.c_void_p] * 15
        lib.dendsn_backward_noalloc.restype = ctypes.c_int
        _noalloc_ready = True
    _check("dendsn_backward_noalloc", lib.dendsn_backward_noalloc(
        ctypes.byref(cfg), _ptr(x), _ptr(alpha), _ptr(xi), _ptr(zeta), _ptr(kappa),
        _ptr(mask), _ptr(grad_spikes), _ptr(grad_v), _ptr(saved), _ptr(grad_x),
        _ptr(grad_alpha), _ptr(grad_xi), _ptr(grad_zeta), _ptr(grad_kappa), _stream(stream)))


# ------------------------------------------------------------------ point-neuron LIF layer
def dendsn_lif_workspace_size(cfg: dendsn_lif_config) -> int:
    """saved_bytes of the LIF layer (checkpoints; 0 for T <= 8)."""
    s = ctypes.c_size_t(0)
    _check("dendsn_lif_workspace_size",
           load().dendsn_lif_workspace_size(ctypes.byref(cfg), ctypes.byref(s)))
    return int(s.value)


def _lif_need(cfg, **tensors):
    sx = 2 if cfg.x_dtype == BF16 else 4
    n = cfg.T * cfg.B * cfg.N
    for name, t in tensors.items():
        if t is None:
            continue
        need = (dendsn_lif_workspace_size(cfg) if name == "saved" else
                n * 4 if name in ("v_out", "grad_v") else n * sx)
        have = t.numel() * t.element_size()
        if have < need:
            raise ValueError(f"{name}: {have} bytes, the config needs {need}")


def dendsn_lif_forward(cfg, x, spikes, v_out=None, saved=None, stream=None):
    _lif_need(cfg, x=x, spikes=spikes, v_out=v_out, saved=saved)
    _check("dendsn_lif_forward", load().dendsn_lif_forward(
        ctypes.byref(cfg), _ptr(x), _ptr(spikes), _ptr(v_out), _ptr(saved), _stream(stream)))


def dendsn_lif_backward(cfg, x, grad_spikes, grad_v, saved, grad_x, stream=None):
    _lif_need(cfg, x=x, grad_spikes=grad_spikes, grad_v=grad_v, saved=saved, grad_x=grad_x)
    _check("dendsn_lif_backward", load().dendsn_lif_backward(
        ctypes.byref(cfg), _ptr(x), _ptr(grad_spikes), _ptr(grad_v), _ptr(saved),
        _ptr(grad_x), _stream(stream)))


def lif_forward(cfg, x, want_v=False, saved=None, stream=None):
    """Allocating LIF forward of x [T, B, N]. Returns (spikes, v or None)."""
    if tuple(x.shape) != (cfg.T, cfg.B, cfg.N) or x.dtype != _xdtype(cfg):
        raise ValueError(f"x must be {_xdtype(cfg)} [{cfg.T},{cfg.B},{cfg.N}]")
    spikes = torch.empty_like(x)
    v = torch.empty(x.shape, dtype=torch.float32, device=x.device) if want_v else None
    dendsn_lif_forward(cfg, x, spikes, v, saved, stream)
    return spikes, v


def lif_backward(cfg, x, grad_spikes, grad_v=None, saved=None, stream=None):
    """Allocating LIF backward. Returns dL/dX with x's shape and dtype."""
    gx = torch.empty_like(x)
    dendsn_lif_backward(cfg, x, grad_spikes, grad_v, saved, gx, stream)
    return gx


def lif_workspace(cfg, device=None):
    """The LIF checkpoint buffer, or None when T <= 8."""
    sb = dendsn_lif_workspace_size(cfg)
    return torch.empty(sb, dtype=torch.uint8, device=device or torch.device("cuda")) if sb else None


# ------------------------------------------------------------------ tensor-level helpers
def _xdtype(cfg) -> torch.dtype:
    return torch.bfloat16 if cfg.x_dtype == BF16 else torch.float32


def _check_shapes(cfg, x, alpha, xi, zeta, kappa, mask):
    T, B, N, K, C, Kb = cfg.T, cfg.B, cfg.N, cfg.K, cfg.C, cfg.K // cfg.G
    if cfg.layout == LAYOUT_PAPER:
        # [T, B, N / inner, K, inner] in any contiguous shape with that element order
        if x.numel() != T * B * N * K or x.dtype != _xdtype(cfg) or x.dim() < 2 or \
                tuple(x.shape[:2]) != (T, B):
            raise ValueError(f"x must be {_xdtype(cfg)} [{T},{B},...] with {T * B * N * K} elements")
    elif tuple(x.shape) != (T, B, N, K) or x.dtype != _xdtype(cfg):
        raise ValueError(f"x must be {_xdtype(cfg)} [{T},{B},{N},{K}], got {x.dtype} {tuple(x.shape)}")
    for name, t, shp in (("alpha", alpha, (C, K)), ("xi", xi, (C, K)), ("zeta", zeta, (C, Kb)),
                         ("kappa", kappa, (C, Kb))):
        if tuple(t.shape) != shp or t.dtype != torch.float32:
            raise ValueError(f"{name} must be float32 {shp}, got {t.dtype} {tuple(t.shape)}")
    if mask is not None:
        rows = N if cfg.mask_per_neuron else C
        if tuple(mask.shape) != (rows, Kb) or mask.dtype != torch.uint8:
            raise ValueError(f"mask must be uint8 [{rows},{Kb}]")


def workspace(cfg, device=None):
    """Allocates (saved, scratch) byte buffers; None where zero bytes are needed."""
    sb, wb = dendsn_workspace_size(cfg)
    dev = device or torch.device("cuda")
    saved = torch.empty(sb, dtype=torch.uint8, device=dev) if sb else None
    scratch = torch.empty(max(wb, 16), dtype=torch.uint8, device=dev)
    return saved, scratch


def forward(cfg, x, alpha, xi, zeta, kappa, mask=None, want_v=False, saved=None, stream=None):
    """Allocating forward. Returns (spikes, v or None)."""
    _check_shapes(cfg, x, alpha, xi, zeta, kappa, mask)
    shape = (cfg.T, cfg.B, cfg.N)
    spikes = torch.empty(shape, dtype=x.dtype, device=x.device)
    v = torch.empty(shape, dtype=torch.float32, device=x.device) if want_v else None
    dendsn_forward(cfg, x, alpha, xi, zeta, kappa, mask, spikes, v, saved, stream)
    return spikes, v


def backward(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v=None, saved=None,
             scratch=None, stream=None, want_beta=False):
    """Allocating backward. Returns dict gx, galpha, gxi, gzeta, gkappa, and with want_beta
    also gbeta (the gradient of a learnable somatic decay, per channel; computed by the
    separate dendsn_backward_plif kernel build)."""
    _check_shapes(cfg, x, alpha, xi, zeta, kappa, mask)
    if scratch is None:
        _, scratch = workspace(cfg, x.device)
    dev = x.device
    C, K, Kb = cfg.C, cfg.K, cfg.K // cfg.G
    out = dict(gx=torch.empty_like(x),
               galpha=torch.empty((C, K), dtype=torch.float32, device=dev),
               gxi=torch.empty((C, K), dtype=torch.float32, device=dev),
               gzeta=torch.empty((C, Kb), dtype=torch.float32, device=dev),
               gkappa=torch.empty((C, Kb), dtype=torch.float32, device=dev))
    grads = (out["gx"], out["galpha"], out["gxi"], out["gzeta"], out["gkappa"])
    if want_beta:
        out["gbeta"] = torch.empty((C,), dtype=torch.float32, device=dev)
        dendsn_backward_plif(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                             *grads, out["gbeta"], scratch, stream)
    else:
        dendsn_backward(cfg, x, alpha, xi, zeta, kappa, mask, grad_spikes, grad_v, saved,
                        *grads, scratch, stream)
    return out


class DendSNFunction(torch.autograd.Function):
    """autograd wrapper: S = DendSN(X; alpha, xi, zeta, kappa[, beta]) (Eq. dendsn).

    alpha may be a scalar tensor (the paper's layer-wide decay) or [C, K]; its gradient is
    reduced to its own shape. The mask is a constant. beta: None (the somatic decay is
    cfg.beta, a constant) or a 0-dim tensor, a learnable decay (PLIF soma); its value
    replaces cfg.beta and its gradient is the sum of the per-channel dL/dbeta.
    """

    @staticmethod
    def forward(ctx, x, alpha, xi, zeta, kappa, mask, cfg, beta=None):
        if beta is not None:
            cfg = dendsn_config.from_buffer_copy(cfg)
            cfg.beta = float(beta)
        a = alpha.expand(cfg.C, cfg.K).contiguous().float()
        saved, scratch = workspace(cfg, x.device)
        s, _ = forward(cfg, x.contiguous(), a, xi.contiguous(), zeta.contiguous(),
                       kappa.contiguous(), mask, saved=saved)
        ctx.cfg = cfg
        ctx.alpha_shape = alpha.shape
        ctx.learn_beta = beta is not None
        ctx.ws = (saved, scratch)
        ctx.save_for_backward(x, a, xi, zeta, kappa, mask)
        return s

    @staticmethod
    def backward(ctx, gs):
        x, a, xi, zeta, kappa, mask = ctx.saved_tensors
        saved, scratch = ctx.ws
        g = backward(ctx.cfg, x, a, xi, zeta, kappa, mask, gs.contiguous().to(x.dtype),
                     None, saved, scratch, want_beta=ctx.learn_beta)
        ga = g["galpha"].sum_to_size(ctx.alpha_shape)
        gb = g["gbeta"].sum() if ctx.learn_beta else None
        return g["gx"], ga, g["gxi"], g["gzeta"], g["gkappa"], None, None, gb
