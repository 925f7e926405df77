"""Seeded synthetic workloads for the PRESTO draft-and-verify step.

This module only draws random inputs with the shapes and value distributions of
the paper's workloads (Qwen3-8B-class target, dFlash-style diffusion drafter,
self-speculative dLLM).  It holds none of the method's arithmetic: no top-k, no
scoring, no tree search, no attention.  Both the CPU oracle and the CUDA path
consume what it returns; neither is imported here.
"""

from .workloads import (  # noqa: F401
    WORKLOADS,
    Workload,
    attention_inputs,
    ctx_tokens,
    drafter_logits,
    frequent_tokens,
    kv_lengths,
    node_paths,
    target_tokens,
    trigram_entries,
)
