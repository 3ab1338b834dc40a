"""Seeded synthetic inputs for the A-PACK inner-LLM prune step.

This package is shared by the tests, the benchmark and the smoke check.  It
holds no arithmetic of the method itself (no attention scores, no selection,
no compaction): only the counter-based random number generator, the token
layouts of the audio-video workloads and the planting of high-relevance keys.

Both the CUDA path and the CPU oracle receive the arrays produced here.
"""

from .gen import (  # noqa: F401
    TID_Q, TID_K, TID_V, TID_HIDDEN, TID_PLANT, TID_RAGGED, TID_POS,
    splitmix64, hash_stream, normal_bf16_bits, uniform_u32,
    bf16_bits_to_f32, f32_to_bf16_bits,
)
from .configs import Workload, SeqLayout, workload, WORKLOADS  # noqa: F401
