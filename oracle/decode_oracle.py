"""CPU oracle of the decode-step attention over a (compacted) KV cache
(test infrastructure only).

TEST INFRASTRUCTURE: only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` leg of ``bench.py`` may use it; it shares no code with the
CUDA path.

Sec. 3.2 (last sentence) and App. G ("decoding throughput"): after pruning,
every autoregressive decode step attends from its one new query token to the
shortened cache of each layer.  What one layer's attention computes for that
token, per sequence b and query head h (key head g = h // (Hq / Hkv), the
grouped-query convention used throughout):

    out[b, h] = sum_j softmax_j(q[b, h] . k[j, g] / sqrt(D)) v[j, g],

over every cached token j of the sequence (the decode token attends to the
whole cache, multimodal or not).  fp64 from exactly widened bf16; numpy's
matmul and exp are the only library steps.
"""

import numpy as np

from .apack_oracle import bf16_to_f64


def decode_attention(q_bits, k_bits, v_bits, cu_seqlens, num_q_heads, num_kv_heads):
    """q_bits: uint16 [B, Hq, D]; k_bits, v_bits: uint16 [T, Hkv, D], packed by
    cu_seqlens [B+1].  Returns float64 [B, Hq, D]; a sequence with an empty
    cache gets zeros."""
    q = bf16_to_f64(q_bits)
    k = bf16_to_f64(k_bits)
    v = bf16_to_f64(v_bits)
    B = len(cu_seqlens) - 1
    D = q.shape[2]
    group = num_q_heads // num_kv_heads
    out = np.zeros((B, num_q_heads, D))
    for b in range(B):
        lo, hi = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
        if hi == lo:
            continue
        for h in range(num_q_heads):
            g = h // group
            x = k[lo:hi, g, :] @ q[b, h] / np.sqrt(D)
            p = np.exp(x - x.max())
            p /= p.sum()
            out[b, h] = p @ v[lo:hi, g, :]
    return out
