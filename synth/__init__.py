"""Seeded synthetic inputs for the Early-Bird decoding step.

This package is the one piece of code that both the CUDA path (through its
Python binding) and the CPU oracle consume.  It holds none of the method's
arithmetic: it only draws random tensors, bf16-rounds them, lays out the
router parameter list, and describes the workload shapes.
"""
from .configs import (Shape, SHAPES, tiny, llada, dream, loop_shape, loop_tiny,
                      llada_full, tiny_full, loop_full_tiny, loop_full,
                      sweep_points, sweep_point)
from .gen import (StepInputs, make_step_inputs, normal_f32, normal_bf16,
                  uniform01, bf16_round, bf16_to_f32, f32_to_bf16_bits,
                  preset_in_block, loop_window_inputs, loop_kv, window_sizes,
                  with_suffix_cache, MASK_TOKEN)
from .router_init import (RouterLayout, router_layout, router_weights,
                          splitmix64_uniform, pack_blob, unpack_blob)

__all__ = [
    "Shape", "SHAPES", "tiny", "llada", "dream", "loop_shape", "loop_tiny",
    "llada_full", "tiny_full", "loop_full_tiny", "loop_full",
    "sweep_points", "sweep_point", "StepInputs", "make_step_inputs",
    "normal_f32", "normal_bf16", "uniform01", "bf16_round", "bf16_to_f32",
    "f32_to_bf16_bits", "preset_in_block", "loop_window_inputs", "loop_kv",
    "window_sizes", "with_suffix_cache",
    "MASK_TOKEN", "RouterLayout", "router_layout", "router_weights",
    "splitmix64_uniform", "pack_blob", "unpack_blob",
]
