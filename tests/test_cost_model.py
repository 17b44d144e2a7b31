"""The roofline cost model of the benchmark, counted by hand for a few layers.

Bytes per neuron-step (x, spikes, grad_spikes and grad_x in the layer's dtype):
  forward  K s + s        (read x, write S)
  backward K s + s + K s  (re-read x, read dL/dS, write dL/dX)

Float32 operations per neuron-step (a fused multiply-add counts once), Mexican hat, G = 1,
Stateful, hard reset, no residual, K = 4:
  forward   V^d 4 + u 4 + u^2 4 + psi 2 x 4 + kappa*m sum 4 + charge and threshold 2 = 26
  backward  recompute 26 + u and u^2 again 8 + soma adjoint 7
            + per branch (dL/dY 1, psi' 5, dr/du 1, dzeta 2, dkappa 2) x 4 = 44
            + per compartment (dL/dV^d 1, dxi 1, scan 1, dalpha 1) x 4 = 16        -> 101
  special-function unit: forward one exp2 per branch (4); backward the recompute's 4, the
  surrogate's reciprocal and the reverse step's exp2 per branch: 9 (the kernels' measured
  XU-pipe instructions per neuron-step: 4.5 and 9.5)
"""
import pytest

from paper_2412_06355_gb300.workloads import WORKLOADS


@pytest.mark.parametrize("name, fwd, bwd", [
    ("conv", 20, 36),               # K = 4 float32
    ("deepconv_bf16", 18, 34),      # K = 8 bf16
    ("token_dbg", 36, 68),          # K = 8 float32
])
def test_algorithmic_bytes_per_neuron_step(name, fwd, bwd):
    w = WORKLOADS[name]
    ab = w.algorithmic_bytes()
    assert ab["forward"] == fwd * w.neuron_steps
    assert ab["backward"] == bwd * w.neuron_steps
    assert ab["total"] == (fwd + bwd) * w.neuron_steps


def test_fp32_ops_mexican_hat_conv():
    ops = WORKLOADS["conv"].fp32_ops_per_neuron_step()
    assert (ops["forward"], ops["backward"]) == (26, 101)
    assert ops["sfu"] == {"forward": 4, "backward": 9}


def test_fp32_ops_variants():
    w = WORKLOADS["conv"]
    # identity branch, G = 1: r = |u| (no square, no psi arithmetic, no psi')
    #   forward 4 + 4 + 4 + 2 = 14; backward 14 + 4 + 7 + (1 + 1 + 2 + 2) x 4 + 16 = 65
    ops = w.with_(psi="identity").fp32_ops_per_neuron_step()
    assert (ops["forward"], ops["backward"]) == (14, 65)
    assert ops["sfu"] == {"forward": 0, "backward": 1}
    # Stateless: no V^d recursion, no reverse scan, no dalpha
    #   forward 26 - 4 = 22; backward 22 + 8 + 7 + 44 + 2 x 4 = 89
    ops = w.with_(stateless=True).fp32_ops_per_neuron_step()
    assert (ops["forward"], ops["backward"]) == (22, 89)
    # soft reset: one more operation (V^s - theta) in the charge
    assert w.with_(reset="soft").fp32_ops_per_neuron_step()["forward"] == 27
    # two compartments per branch (K = 4, Kb = 2), Mexican hat: psi and the sums per branch,
    # dr/du per compartment; psi'(r)/r = (r^2 - 3) e needs no 1/r
    #   forward 4 + 4 + 4 + (2 + 1) x 2 + 2 = 20; backward 20 + 8 + 7 + 10 x 2 + 4 + 16 = 75
    ops = w.with_(G=2).fp32_ops_per_neuron_step()
    assert (ops["forward"], ops["backward"]) == (20, 75)
    assert ops["sfu"] == {"forward": 2, "backward": 5}
    # two compartments per branch, identity: r = sqrt(r^2) forward, 1/r backward (SFU), and
    # the product dL/dr / r per branch
    #   forward 4 + 4 + 4 + 2 + 2 = 16; backward 16 + 8 + 7 + 5 x 2 + (4 + 2) + 16 = 63
    ops = w.with_(G=2, psi="identity").fp32_ops_per_neuron_step()
    assert (ops["forward"], ops["backward"]) == (16, 63)
    assert ops["sfu"] == {"forward": 2, "backward": 5}
