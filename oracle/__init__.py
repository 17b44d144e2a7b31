"""CPU float64 oracle of the DendSN layer: TEST INFRASTRUCTURE ONLY.

Only the tests, the smoke check and the benchmark's CPU-baseline leg may import
this package. The product path (the CUDA library and its binding) never does.
"""
from .oracle import (OracleConfig, build, forward, backward, layer_channels,
                     forward_layer, backward_layer, layer_x, layer_gx, to_f64,
                     LIFConfig, lif_forward, lif_backward)

__all__ = ["OracleConfig", "build", "forward", "backward", "layer_channels",
           "forward_layer", "backward_layer", "layer_x", "layer_gx", "to_f64",
           "LIFConfig", "lif_forward", "lif_backward"]
