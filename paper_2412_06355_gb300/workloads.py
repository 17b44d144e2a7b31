"""Seeded synthetic inputs for the DendSN layer (forward + BPTT backward).

This module only draws random tensors with the shapes and value distributions of
the layer workloads; it holds none of the neuron's arithmetic. Both the CUDA path
and the CPU oracle are fed from it, so they see identical bits.

Layout (the library's ABI):
  x      [T, B, N, K]   branch/compartment input currents, K innermost; or, for
                        layout "paper", [T, B, N / inner, K, inner]: a conv layer's
                        output read as (C_o, P, H, W) with inner = H * W
  alpha  [C, K]         compartment decay factors           (Eq. methods-compartment)
  xi     [C, K]         translation factors                 (Eq. methods-branch-aggregation)
  zeta   [C, Kb]        dilation factors, Kb = K / G        (Eq. methods-branch-aggregation)
  kappa  [C, Kb]        branch strengths                    (Eq. methods-soma-input)
  mask   [C, Kb] or [N, Kb] uint8 branch-gating mask        (Eq. methods-dbg-mask / -sampling)
  gs     [T, B, N]      upstream gradient w.r.t. the spikes
  gv     [T, B, N]      upstream gradient w.r.t. the somatic potential (optional)

Neuron n of a sample belongs to parameter channel c(n) = (n // inner) % C, so
neurons at the spatial positions of one conv channel share a parameter set
(Methods, "Dendritic spiking neural networks", constraint 3).

Draw order is fixed: x, alpha, xi, zeta, kappa, mask, gs, gv, all from one
torch.Generator seeded with the workload's seed.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int
    B: int
    N: int
    K: int
    G: int
    C: int
    inner: int
    dtype: str          # "f32" or "bf16": dtype of x, spikes, gs and gx
    psi: str            # "mh" (Mexican hat, Eq. methods-mexican-hat) or "identity"
    reset: str          # "hard" (Eq. methods-lif-reset-charge) or "soft"
    theta: float = 1.0
    beta: float = 0.5
    x_mean: float = 0.3
    x_std: float = 1.0
    x_density: float = 1.0        # fraction of nonzero inputs (event-stream layer: 0.2)
    mask_p: Optional[float] = None  # Bernoulli(p) branch mask; None = no mask
    mask_per_neuron: bool = False
    stateless: bool = False
    residual: bool = False
    detach_reset: bool = False
    layout: str = "kinner"          # "kinner" [T,B,N,K] or "paper" [T,B,N/inner,K,inner]
    seed: int = 0

    @property
    def Kb(self) -> int:
        return self.K // self.G

    @property
    def neurons(self) -> int:
        return self.B * self.N

    @property
    def neuron_steps(self) -> int:
        return self.T * self.B * self.N

    @property
    def x_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    def algorithmic_bytes(self) -> dict:
        """Bytes a fused forward+backward must move per step, by kernel.

        forward : read x (K elements) + write spikes (1 element) per neuron-step
        backward: re-read x (K) + read gs (1) + write gx (K) per neuron-step
        Parameters and the mask (< 1 MB, cache-resident) are not counted.
        """
        ns, s = self.neuron_steps, self.x_bytes
        fwd = ns * (self.K * s + s)
        bwd = ns * (self.K * s + s + self.K * s)
        return {"forward": fwd, "backward": bwd, "total": fwd + bwd}

    def fp32_ops_per_neuron_step(self) -> dict:
        """Float32 arithmetic a fused forward+backward needs per neuron-step, by kernel: a
        cost model counted from the equations (a fused multiply-add is one operation; 1/zeta
        and -xi/zeta are folded into the parameters once; exp2, sqrt and 1/x run on the
        special-function unit and are counted apart, in `sfu`). Address arithmetic, loads,
        stores, conversions, selects and compares other than the threshold are the
        implementation's, not counted.

        forward: per compartment V^d (Eq. methods-compartment; none when Stateless),
        u = V^d/zeta - xi/zeta and its square (Eq. methods-branch-aggregation; for G = 1 the
        identity branch needs only |u|, for G > 1 it takes a square root), the residual
        term; per branch psi (Mexican hat: the exponent's scale and (1 - r^2) e, Eq.
        methods-mexican-hat) and the kappa*m sum (Eq. methods-soma-input); per neuron the
        charge and the threshold (+1 for the soft reset).
        backward: the forward's recompute, then the reverse step: u and r^2 again; the soma
        adjoint (dV[t+1]/dS, dL/dS, the surrogate's argument, square and + 1, dL/dV^s: 7,
        Eq. methods-sg); per branch dL/dY, psi' (Mexican hat: the exponent's scale, y,
        r^2 - 3, two products: 5; psi'(r)/r needs no 1/r), dr/du (G = 1: one product per
        branch; G > 1: one per compartment, plus 1/r and a product per branch for the
        identity), dzeta (2) and dkappa (2); per compartment dL/dV^d, dxi, the residual
        gradient, and (Stateful) the reverse scan and dalpha.
        """
        K, Kb, G = self.K, self.Kb, self.G
        mh = self.psi == "mh"
        stateful = not self.stateless
        square = K if (mh or G > 1) else 0
        fwd = ((K if stateful else 0) + K + square + (K if self.residual else 0)
               + Kb * ((2 if mh else 0) + 1)
               + 2 + (1 if self.reset == "soft" else 0))
        drdu = Kb if G == 1 else K + (0 if mh else Kb)
        rev = (K + square + 7 + Kb * (1 + (5 if mh else 0) + 2 + 2) + drdu
               + K * (1 + 1 + (2 if stateful else 0)) + (K if self.residual else 0))
        sfu_f = Kb if (mh or G > 1) else 0
        sfu_b = sfu_f + 1 + (Kb if (mh or G > 1) else 0)
        return {"forward": fwd, "backward": fwd + rev,
                "sfu": {"forward": sfu_f, "backward": sfu_b}}

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The layer shapes: a tiny case, a conv layer (also in the paper's (C_o, P, H, W) layout
# with two compartments per branch), a deeper bf16 conv layer, a long-horizon
# event-stream layer with sparse input, a transformer-token layer with per-neuron branch
# gating, and two T = 2048 cases.
WORKLOADS = {
    "tiny": Workload("tiny", T=4, B=2, N=64, K=4, G=1, C=64, inner=1, dtype="f32",
                     psi="mh", reset="hard", seed=0),
    "conv": Workload("conv", T=4, B=64, N=131072, K=4, G=1, C=128, inner=1024,
                     dtype="f32", psi="mh", reset="hard", seed=1),
    "deepconv_bf16": Workload("deepconv_bf16", T=8, B=128, N=65536, K=8, G=1, C=256,
                              inner=256, dtype="bf16", psi="mh", reset="soft", seed=2),
    "event": Workload("event", T=64, B=32, N=131072, K=4, G=1, C=128, inner=1024,
                      dtype="f32", psi="mh", reset="hard", x_mean=0.8, x_std=1.0,
                      x_density=0.2, seed=3),
    "conv_paper_p4b2": Workload("conv_paper_p4b2", T=4, B=64, N=131072, K=4, G=2, C=128,
                                inner=1024, dtype="f32", psi="mh", reset="hard",
                                layout="paper", seed=5),
    "token_dbg": Workload("token_dbg", T=4, B=64, N=196 * 384, K=8, G=1, C=384, inner=1,
                          dtype="f32", psi="mh", reset="hard", mask_p=0.5,
                          mask_per_neuron=True, seed=4),
    # long horizon: the L5PC fitting setting (one neuron with P = 4 compartments on
    # B = 2 branches, T = 2048, batch 16, beta = 0.95; Methods "Details of L5PC
    # approximation" and the hyperparameter table), and the same horizon on a layer
    "l5pc": Workload("l5pc", T=2048, B=16, N=1, K=4, G=2, C=1, inner=1, dtype="f32",
                     psi="mh", reset="hard", beta=0.95, x_mean=0.1, x_std=0.5,
                     x_density=0.3, seed=6),
    "long_t": Workload("long_t", T=2048, B=16, N=4096, K=4, G=2, C=4, inner=1024,
                       dtype="f32", psi="mh", reset="hard", beta=0.95, x_mean=0.1,
                       x_std=0.5, x_density=0.3, seed=7),
}


def torch_dtype(w: Workload) -> torch.dtype:
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32


def make_inputs(w: Workload, device: str = "cpu", with_gv: bool = False) -> dict:
    """Draw every input of one forward+backward step of workload `w`.

    Value distributions: x ~ N(x_mean, x_std) (times Bernoulli(x_density) when
    sparse), alpha ~ U(0.5, 0.95), xi ~ N(0, 0.1), zeta ~ U(0.8, 1.2),
    kappa ~ N(1/K, 0.1), mask ~ Bernoulli(mask_p), gs ~ N(0, 1), gv ~ N(0, 1).
    x, gs are rounded to the workload dtype; parameters stay float32.
    """
    g = torch.Generator(device=device)
    g.manual_seed(w.seed)
    f32 = dict(dtype=torch.float32, device=device)
    T, B, N, K, C, Kb = w.T, w.B, w.N, w.K, w.C, w.Kb
    x = torch.randn((T, B, N, K), generator=g, **f32).mul_(w.x_std).add_(w.x_mean)
    if w.x_density < 1.0:
        keep = torch.rand((T, B, N, K), generator=g, **f32) < w.x_density
        x.mul_(keep)
        del keep
    x = x.to(torch_dtype(w))
    if w.layout == "paper":
        x = to_paper_layout(x, w.inner)
    alpha = torch.rand((C, K), generator=g, **f32).mul_(0.45).add_(0.5)
    xi = torch.randn((C, K), generator=g, **f32).mul_(0.1)
    zeta = torch.rand((C, Kb), generator=g, **f32).mul_(0.4).add_(0.8)
    kappa = torch.randn((C, Kb), generator=g, **f32).mul_(0.1).add_(1.0 / K)
    mask = None
    if w.mask_p is not None:
        rows = N if w.mask_per_neuron else C
        mask = (torch.rand((rows, Kb), generator=g, **f32) < w.mask_p).to(torch.uint8)
    gs = torch.randn((T, B, N), generator=g, **f32).to(torch_dtype(w))
    gv = torch.randn((T, B, N), generator=g, **f32) if with_gv else None
    return dict(x=x, alpha=alpha, xi=xi, zeta=zeta, kappa=kappa, mask=mask, gs=gs, gv=gv)


def make_lif_inputs(T: int, B: int, N: int, dtype: str = "f32", seed: int = 0,
                    device: str = "cpu", with_gv: bool = False, x_mean: float = 0.5,
                    x_std: float = 1.0) -> dict:
    """Inputs of the point-neuron LIF layer: x ~ N(x_mean, x_std) [T, B, N] (one current
    per neuron), gs ~ N(0, 1) [T, B, N] in the layer dtype, gv ~ N(0, 1) float32.
    Draw order x, gs, gv from one generator."""
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    f32 = dict(dtype=torch.float32, device=device)
    dt = torch.bfloat16 if dtype == "bf16" else torch.float32
    x = torch.randn((T, B, N), generator=g, **f32).mul_(x_std).add_(x_mean).to(dt)
    gs = torch.randn((T, B, N), generator=g, **f32).to(dt)
    gv = torch.randn((T, B, N), generator=g, **f32) if with_gv else None
    return dict(x=x, gs=gs, gv=gv)


def to_paper_layout(x: torch.Tensor, inner: int) -> torch.Tensor:
    """[T, B, N, K] -> the paper's [T, B, N / inner, K, inner] (a pure permutation)."""
    T, B, N, K = x.shape
    return x.reshape(T, B, N // inner, inner, K).permute(0, 1, 2, 4, 3).contiguous()


def from_paper_layout(x: torch.Tensor, N: int, K: int, inner: int) -> torch.Tensor:
    """The paper's [T, B, N / inner, K, inner] -> [T, B, N, K] (a pure permutation)."""
    T, B = x.shape[:2]
    return x.reshape(T, B, N // inner, K, inner).permute(0, 1, 2, 4, 3).reshape(T, B, N, K)


def scaled(w: Workload, B: Optional[int] = None, N: Optional[int] = None,
           T: Optional[int] = None) -> Workload:
    """Same layer kind at a smaller size (for oracle-sized parity runs).

    N must stay a multiple of C * inner so the channel map is unchanged.
    """
    kw = {}
    if B is not None:
        kw["B"] = B
    if N is not None:
        if N % (w.C * w.inner) != 0:
            raise ValueError("N must be a multiple of C*inner")
        kw["N"] = N
    if T is not None:
        kw["T"] = T
    return w.with_(**kw)
