"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle."""
from .layers import (BLOCK_LLAMA2_7B, CONFIGS, Layer, block_hessians, block_layers,
                     config_layer, rtn_host_np, rtn_host_torch, small_layer, tiny_layer)

__all__ = ["BLOCK_LLAMA2_7B", "CONFIGS", "Layer", "block_hessians", "block_layers",
           "config_layer", "rtn_host_np", "rtn_host_torch", "small_layer", "tiny_layer"]
