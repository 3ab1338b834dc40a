"""CPU oracle of the A-PACK inner-LLM prune step (test infrastructure only).

Only the tests, the smoke check and the CPU-baseline leg of the benchmark may
import this package.  The CUDA library never calls it, and it never calls the
CUDA library: the two share no code.  See ``apack_oracle.py``.
"""

from .prellm_oracle import frame_embeddings, window_cka, gate, frame_alignment  # noqa: F401
from .decode_oracle import decode_attention  # noqa: F401
from .apack_oracle import (  # noqa: F401
    MOD_OTHER, MOD_AUDIO, MOD_VISUAL, SOFTMAX_MM, SOFTMAX_CAUSAL_ROW,
    bf16_to_f64, relevance_scores, keep_count, step_keep_counts, select_keep,
    compact_rows, new_cu_seqlens, prune_step, score_tolerance,
)
