"""The kernels' exponential and reciprocal approximations, read through the C ABI.

The Mexican hat psi(r) = (1 - r^2) e^{-r^2/2} (Eq. methods-mexican-hat), its derivative
psi'(r) = r (r^2 - 3) e^{-r^2/2} and the arctan surrogate's derivative
sg(x) = 1 / (1 + pi^2 x^2) (Eq. methods-sg) are evaluated on the GPU with the hardware
2^x and 1/x approximations (e^{-r^2/2} = 2^{-r^2 log2(e) / 2}). Each is read out of an
existing output on a layer that reduces the neuron to that one function:
  psi      K = 1, T = 1, alpha = xi = 0, zeta = kappa = 1, no spike: V^s[0] = psi(x)
  psi'     the same layer's backward with dL/dS = 0, dL/dV^s = 1: dL/dX[0] = psi'(x)
  sg       identity branch, theta = 0, dL/dS = 1: dL/dX[0] = sg(x) for x > 0
over a dense grid of float32 inputs (r in [-8, 8], x in (0, 10]), and compared with
float64 values of the same functions at the same float32 inputs.

Each error is bounded by a first-order model of the float32 evaluation with unit
roundoff u = 2^-24 and a relative error eps_e of the hardware 2^x of at most 2^-21:
  psi   e [ |1 - r^2| (eps_e + |s| ln2 u + 2u) + r^2 u (1 + |1 - r^2| / 2) ] + u |psi|,
        s = -r^2 log2(e) / 2 (the exponent; its rounding moves e by |s| ln2 u relative)
  psi'  |r| e [ |r^2 - 3| (eps_e + |s| ln2 u + 3u) + r^2 u ]
  sg    relative (3u + eps_r) with eps_r = 2^-22 for the hardware 1/x
and the test requires every error within twice its model. With DENDSN_PARITY_REPORT set,
the worst error over the model and the largest relative errors are written there.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

from paper_2412_06355_gb300 import binding

pytestmark = pytest.mark.gpu

U = 2.0 ** -24
EPS_EXP2 = 2.0 ** -21
EPS_RCP = 2.0 ** -22
LN2 = math.log(2.0)
LOG2E = 1.0 / LN2


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.fail("these tests need a CUDA device")
    binding.load()


def point_layer(x: torch.Tensor, psi: str, theta: float):
    """T = 1, one sample, one compartment per neuron, one parameter channel."""
    n = x.numel()
    cfg = binding.make_config(1, 1, n, 1, 1, 1, 1, "f32", psi, "hard", theta=theta, beta=0.5)
    one = torch.ones((1, 1), device="cuda")
    zero = torch.zeros((1, 1), device="cuda")
    return cfg, x.reshape(1, 1, n, 1).contiguous(), (zero, zero.clone(), one, one.clone())


def _report(name, stats):
    out = os.environ.get("DENDSN_PARITY_REPORT")
    if out:
        os.makedirs(out, exist_ok=True)
        with open(os.path.join(out, f"transcendental_{name}.json"), "w") as f:
            json.dump(stats, f, indent=1)
    print(name, json.dumps(stats))


def _grid(lo, hi, n):
    return torch.linspace(lo, hi, n, dtype=torch.float32)


def test_mexican_hat_and_its_derivative():
    x = torch.cat([_grid(-8.0, 8.0, 1 << 20), torch.tensor([0.0, 1.0, -1.0, 3.0 ** 0.5])])
    x = x[: (x.numel() // 4) * 4]
    cfg, xd, prm = point_layer(x.cuda(), "mh", theta=1e30)
    s, v = binding.forward(cfg, xd, *prm, None, want_v=True)
    gs = torch.zeros((1, 1, x.numel()), device="cuda")
    gv = torch.ones((1, 1, x.numel()), device="cuda")
    g = binding.backward(cfg, xd, *prm, None, gs, gv)
    torch.cuda.synchronize()
    assert torch.count_nonzero(s).item() == 0
    r = x.double().numpy()
    e = np.exp(-0.5 * r * r)
    sx = np.abs(-0.5 * LOG2E * r * r)
    psi = (1.0 - r * r) * e
    dpsi = r * (r * r - 3.0) * e
    got_psi = v.reshape(-1).double().cpu().numpy()
    got_dpsi = g["gx"].reshape(-1).double().cpu().numpy()
    m_psi = e * (np.abs(1 - r * r) * (EPS_EXP2 + sx * LN2 * U + 2 * U)
                 + r * r * U * (1 + np.abs(1 - r * r) / 2)) + U * np.abs(psi)
    m_dpsi = np.abs(r) * e * (np.abs(r * r - 3) * (EPS_EXP2 + sx * LN2 * U + 3 * U) + r * r * U)
    err_psi, err_dpsi = np.abs(got_psi - psi), np.abs(got_dpsi - dpsi)
    # exact special values: psi(0) = 1, psi'(0) = 0
    assert got_psi[r == 0].tolist() and all(v == 1.0 for v in got_psi[r == 0])
    assert all(v == 0.0 for v in got_dpsi[r == 0])
    away = np.abs(np.abs(r) - 1.0) > 0.05            # relative error away from the hat's root
    away_d = (np.abs(np.abs(r) - 3.0 ** 0.5) > 0.05) & (np.abs(r) > 1e-3)
    core, core_d = away & (np.abs(r) <= 4.0), away_d & (np.abs(r) <= 4.0)
    stats = {
        "points": int(r.size),
        "psi_max_err_over_model": float((err_psi / m_psi).max()),
        "psi_max_abs_err": float(err_psi.max()),
        "psi_max_rel_err_r_le_4": float((err_psi[core] / np.abs(psi[core])).max()),
        "psi_max_rel_err_r_le_8": float((err_psi[away] / np.abs(psi[away])).max()),
        "dpsi_max_err_over_model": float((err_dpsi[r != 0] / m_dpsi[r != 0]).max()),
        "dpsi_max_abs_err": float(err_dpsi.max()),
        "dpsi_max_rel_err_r_le_4": float((err_dpsi[core_d] / np.abs(dpsi[core_d])).max()),
        "dpsi_max_rel_err_r_le_8": float((err_dpsi[away_d] / np.abs(dpsi[away_d])).max()),
    }
    _report("mexican_hat", stats)
    assert np.all(err_psi <= 2 * m_psi), stats
    assert np.all(err_dpsi <= 2 * m_dpsi), stats


def test_arctan_surrogate_derivative():
    x = _grid(0.0, 10.0, (1 << 20) + 1)[1:]                 # x > 0: the identity branch's sign is 1
    cfg, xd, prm = point_layer(x.cuda(), "identity", theta=0.0)
    gs = torch.ones((1, 1, x.numel()), device="cuda")
    g = binding.backward(cfg, xd, *prm, None, gs, None)
    torch.cuda.synchronize()
    xx = x.double().numpy()
    sg = 1.0 / (1.0 + math.pi ** 2 * xx * xx)
    got = g["gx"].reshape(-1).double().cpu().numpy()
    rel = np.abs(got - sg) / sg
    model = 3 * U + EPS_RCP
    stats = {"points": int(xx.size), "sg_max_rel_err": float(rel.max()),
             "sg_max_err_over_model": float((rel / model).max()), "model_rel": model}
    _report("surrogate", stats)
    assert np.all(rel <= 2 * model), stats
