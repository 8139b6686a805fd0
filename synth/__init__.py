"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle."""
from .activations import (ACT_CONFIGS, activations_np, activations_torch, config_activations,
                          integer_activations_np)
from .layers import (BLOCK_LLAMA2_7B, CONFIGS, Layer, block_hessians, block_layers,
                     config_layer, rtn_host_np, rtn_host_torch, small_layer, tiny_layer)

__all__ = ["ACT_CONFIGS", "activations_np", "activations_torch", "config_activations",
           "integer_activations_np", "BLOCK_LLAMA2_7B", "CONFIGS", "Layer", "block_hessians", "block_layers",
           "config_layer", "rtn_host_np", "rtn_host_torch", "small_layer", "tiny_layer"]
