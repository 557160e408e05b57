"""Seeded synthetic inputs shaped like the paper's workloads.

This package holds input generation only: random tensors, ragged offsets and
budgets.  It contains none of the method's arithmetic (no softmax, no score
aggregation, no selection), and both the oracle-side tests and the CUDA-side
tests/benchmark draw their inputs from it.
"""
from .synth import (Workload, bf16_bits_to_f32, config, custom, f32_to_bf16_bits,
                    query_rows, CONFIG_NAMES)

__all__ = ["Workload", "bf16_bits_to_f32", "config", "custom", "f32_to_bf16_bits",
           "query_rows", "CONFIG_NAMES"]
