"""CPU oracle of the SGD-KV compression step (test infrastructure; see sgdkv_oracle)."""
from .sgdkv_oracle import (GREEDY, PROPORTIONAL, THRESHOLD, REVERSE, allocate_budgets,
                           mix_head_scores, window_scores,
                           max_pool, select_indices, gather, compress_layer, normalise,
                           decode_attention,
                           bf16_bits_to_f64)
