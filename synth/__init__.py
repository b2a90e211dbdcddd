"""Seeded synthetic inputs for the Similarity Chunk Rolling prefill path.

This package holds only input synthesis (random draws, RoPE applied to the
drawn vectors, rounding to bf16) and the workload table. It contains none of
the method's arithmetic, so that both the CPU oracle and the CUDA path can
consume it without sharing any computation.
"""

from .generate import (  # noqa: F401
    WORKLOADS,
    Workload,
    bf16_bits_to_f32,
    f64_to_bf16_bits,
    generate_layer,
    topic_segments,
    workload,
)
