"""GB300-native (sm_103a) H2O sparse attention: chunked SDPA with summed
attention weights and the H2O cache update, as a C-ABI CUDA library.

The Python layer only marshals torch tensors to the C ABI (include/h2o.h).
"""
from ._binding import (POLICY, H2ODims, H2OError, h2o_backward_workspace_size, h2o_cache_reset,
                       h2o_device_errors, h2o_sdpa_chunk_backward,
                       h2o_sdpa_chunk_backward_lse, h2o_sdpa_chunk_lse,
                       h2o_evict_insert, h2o_evict_insert_q8, h2o_kv_dequantize,
                       h2o_kv_quantize, h2o_kv_replace, h2o_kv_restore, h2o_q8_workspace_size,
                       h2o_scores_add, h2o_sdpa_cache, h2o_sdpa_cache_q8, h2o_sdpa_chunk_q8,
                       h2o_update_q8,
                       h2o_sdpa_chunk, h2o_sdpa_decode_static, h2o_status_string, h2o_update,
                       h2o_update_policy,
                       h2o_version, h2o_workspace_size, load)
from .runner import H2OLayer

__all__ = ["POLICY", "H2ODims", "H2OError", "H2OLayer", "h2o_backward_workspace_size",
           "h2o_cache_reset", "h2o_device_errors", "h2o_sdpa_chunk_backward",
           "h2o_sdpa_chunk_backward_lse", "h2o_sdpa_chunk_lse",
           "h2o_evict_insert", "h2o_evict_insert_q8", "h2o_kv_dequantize", "h2o_kv_quantize",
           "h2o_kv_replace", "h2o_kv_restore", "h2o_q8_workspace_size", "h2o_scores_add",
           "h2o_sdpa_cache", "h2o_sdpa_cache_q8", "h2o_sdpa_chunk", "h2o_sdpa_chunk_q8",
           "h2o_sdpa_decode_static", "h2o_status_string", "h2o_update", "h2o_update_policy",
           "h2o_update_q8", "h2o_version", "h2o_workspace_size", "load"]
