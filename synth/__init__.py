"""Seeded synthetic inputs for LazyMAR's cached decoding step.

This package generates shapes, weights, class labels, decoding orders, token
latents and mask states. It holds none of the method's arithmetic: both the CPU
oracle (through the tests) and the CUDA library (through the tests and the
benchmark) consume what it produces, and neither imports the other.
"""
from .inputs import (  # noqa: F401
    CONFIGS,
    config,
    round_bf16,
    make_weights,
    make_labels,
    make_order,
    make_latent_table,
    mask_counts,
    step_state,
    tiny_state,
    n_compute,
    tensor,
    similarity_inputs,
    distinct_rows,
    HEAD_CONFIGS,
    head_config,
    make_head_weights,
    make_head_noise,
)
