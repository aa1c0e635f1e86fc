"""Seeded synthetic workloads shared by the CUDA path's tests/bench and the oracle."""
from .synth import (PAGE, QWEN3_32B, CONFIG_NAMES, Batch, SparseDraft, config_shape, make_batch,
                    make_config, make_sparse_draft, make_spec_inputs, offsets, philox_uniforms,
                    round_bf16_bits, sigma_for_alpha, draft_len_for_alpha)

__all__ = ["PAGE", "QWEN3_32B", "CONFIG_NAMES", "Batch", "SparseDraft", "config_shape", "make_batch",
           "make_config", "make_sparse_draft", "make_spec_inputs", "offsets", "philox_uniforms",
           "round_bf16_bits", "sigma_for_alpha", "draft_len_for_alpha"]
