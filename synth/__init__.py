"""Seeded synthetic inputs (prompts, weights, workload sizes) for the MBP decode step.

Shared by the CPU oracle and the CUDA path; contains none of the method's arithmetic.
"""
from .configs import (BOUNDARY_BYTE, PAPER, PAPER_MLP, TINY, VOCAB, WORKLOADS, ModelConfig,
                      Workload, gain_for, load_gains, weight_gains)
from .data import (cached_weights, make_weights, param_count, prompt, prompts, round_bf16,
                   tensor_list, words_text, zipf_text)

__all__ = [
    "BOUNDARY_BYTE", "PAPER", "PAPER_MLP", "TINY", "VOCAB", "WORKLOADS", "ModelConfig", "Workload",
    "gain_for", "weight_gains", "load_gains", "cached_weights", "make_weights", "param_count", "prompt", "prompts",
    "round_bf16", "tensor_list", "words_text", "zipf_text",
]
