"""Float64 CPU oracle (test infrastructure only; never on the product path)."""
from .h2o_oracle import (POLICIES, SequenceState, chunk_bounds, lse_merge, run_sequence,
                         sdpa_chunk, update)

__all__ = ["sdpa_chunk", "update", "run_sequence", "SequenceState", "lse_merge", "chunk_bounds",
           "POLICIES"]
