"""GB300-native fused DendSN layer (dendritic spiking neuron, arXiv 2412.06355).

The forward and the BPTT backward of a DendSN layer run as hand-written CUDA
kernels for sm_103a behind the C ABI in include/dendsn.h; `binding` is the thin
Python layer over it and `workloads` draws seeded synthetic layer inputs.
"""
from . import binding, workloads
from .binding import (DendSNError, DendSNFunction, config_of, dendsn_backward, dendsn_forward,
                      dendsn_workspace_size, make_config)

__all__ = ["binding", "workloads", "DendSNError", "DendSNFunction", "config_of",
           "dendsn_backward", "dendsn_forward", "dendsn_workspace_size", "make_config"]
