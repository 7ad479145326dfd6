"""fp64 CPU oracle for the DORA deployment hot path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline legs of
``bench.py`` may import this package.  The CUDA path never does.
"""
from .dora_oracle import *  # noqa: F401,F403
from .dora_oracle import (attention_single, bf16_to_f64, block_attention_half,  # noqa: F401
                          block_mlp_half, compact, cu_from_counts, decode_weights, forward,
                          gather_scores, gelu, layernorm, linear, padded_masked_attention,
                          pruned_block, score_order_key, select_keep, varlen_attention)
