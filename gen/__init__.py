"""Seeded synthetic inputs for the verify / sparsify / state-cache path.

This package only draws random data and lays it out; it contains none of the
arithmetic the method performs on that data (no target softmax, nucleus
filter, accept test, residual, top-k payload or branch selection).  Both the
CUDA path's tests and the CPU oracle's tests read their inputs from here.
"""
from .workloads import (WORKLOADS, Workload, bf16_to_f32, f32_to_bf16, generate, generate_sequences,
                        make_workload)

__all__ = ["WORKLOADS", "Workload", "generate", "generate_sequences", "make_workload", "bf16_to_f32",
           "f32_to_bf16"]
