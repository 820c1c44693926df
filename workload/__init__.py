"""Seeded synthetic workloads shared by the tests, the smoke check and the benchmark.

This package only *draws numbers* (model dimensions, random weights, token ids,
upstream gradients).  It holds none of the method's arithmetic: both the CPU
oracle and the CUDA path receive what it produces as plain arrays.
"""
from .synth import (  # noqa: F401
    PRESETS, TARGETS, ModelDims, preset, tiny, linear_shapes, block_weights,
    embedding, lora_weights, hidden_input, token_ids, upstream_grad, torch_block_weights,
    torch_embedding,
)
