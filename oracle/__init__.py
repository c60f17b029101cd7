"""Float64 CPU oracle (test infrastructure only; never on the product path)."""
from .h2o_oracle import (POLICIES, SequenceState, chunk_bounds, evict_insert, lse_merge,
                         run_sequence, scores_add, sdpa_cache, sdpa_chunk, step_paper_order,
                         update)
from .backward import sdpa_chunk_backward
from .quant import (dequantize_rows, evict_insert_q8, quantize_rows, round_to_bf16, sdpa_cache_q8,
                    sdpa_chunk_q8, update_q8)
from .replay import kv_replace, kv_restore

__all__ = ["sdpa_chunk", "update", "run_sequence", "SequenceState", "lse_merge", "chunk_bounds",
           "POLICIES", "sdpa_cache", "evict_insert", "scores_add", "step_paper_order",
           "kv_replace", "kv_restore", "sdpa_chunk_backward", "quantize_rows", "dequantize_rows",
           "round_to_bf16", "sdpa_cache_q8", "sdpa_chunk_q8", "evict_insert_q8", "update_q8"]
