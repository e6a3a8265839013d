"""Seeded synthetic workloads for the KVLink linked prefill.

This package only draws inputs: workload shapes, document lengths, which pool
documents each query retrieves, and N(0,1) bf16 tensors.  It holds none of the
method's arithmetic (no RoPE, no position bookkeeping, no attention), so both
the fp64 oracle and the CUDA path can take their inputs from it without
sharing any code with each other.
"""
from .configs import CONFIGS, WorkloadConfig, get_config
from .draw import (
    Batch,
    draw_batch,
    normal_bf16,
    f32_to_bf16_bits,
    bf16_bits_to_f32,
    pool_kv,
    fresh_qkv,
    cache_block_tables,
    normal_bf16_torch,
)

__all__ = [
    "CONFIGS",
    "WorkloadConfig",
    "get_config",
    "Batch",
    "draw_batch",
    "normal_bf16",
    "f32_to_bf16_bits",
    "bf16_bits_to_f32",
    "pool_kv",
    "fresh_qkv",
    "cache_block_tables",
    "normal_bf16_torch",
]
