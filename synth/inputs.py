"""Host-side construction of the seeded inputs of a workload.

Arrays are bf16 bit patterns (uint16) so that every consumer widens them the
same exact way.  Q and K of a pruning layer carry the relevance plants; bulk
K/V planes of the other layers are plain draws of the same streams (the CUDA
twin in ``fill.cu`` writes those on the device without a host round trip).
"""

import numpy as np

from .configs import Workload, MOD_AUDIO, MOD_VISUAL
from .gen import (TID_Q, TID_K, TID_V, TID_HIDDEN, TID_PLANT, TID_POS,
                  normal_bf16_bits, hash_stream, uniform_u32, f32_to_bf16_bits,
                  bf16_bits_to_f32, NORMAL_SCALE_F32)


def normal_bf16_at(seed, tid, index):
    """bf16 bits of stream (seed, tid) at arbitrary element indices."""
    index = np.asarray(index, dtype=np.uint64).ravel()
    h = hash_stream(seed, tid, index)
    s = ((h & np.uint64(0xFFFF)) + ((h >> np.uint64(16)) & np.uint64(0xFFFF))
         + ((h >> np.uint64(32)) & np.uint64(0xFFFF)) + (h >> np.uint64(48)))
    z = (s.astype(np.int64) - 131070).astype(np.float32) * NORMAL_SCALE_F32
    return f32_to_bf16_bits(z)


def query_rows(wl: Workload, layer: int) -> np.ndarray:
    """Q of the query span at ``layer``: uint16 [sum n_q, Hq, D]."""
    nq = int(wl.cu_qlens()[-1])
    n = nq * wl.num_q_heads * wl.head_dim
    return normal_bf16_bits(wl.seed, TID_Q + layer, 0, n).reshape(nq, wl.num_q_heads, wl.head_dim)


def planted_tokens(wl: Workload):
    """Global token indices and shift amplitudes of the planted keys.

    Within each sequence the tokens of a modality are ranked by a hash of
    their index; plant entries of that modality take consecutive runs of
    that ranking, so plant sets are disjoint and seed-determined."""
    cu = wl.cu_seqlens()
    mod = wl.modality()
    tok, amp = [], []
    for s, plants in enumerate(wl.plants):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        taken = {MOD_AUDIO: 0, MOD_VISUAL: 0}
        for p in plants:
            cand = np.nonzero(mod[t0:t1] == p.modality)[0]
            h = uniform_u32(wl.seed, TID_PLANT + s, cand)
            order = cand[np.lexsort((cand, h))]
            pick = order[taken[p.modality]:taken[p.modality] + p.count]
            taken[p.modality] += p.count
            tok.append(pick + t0)
            amp.append(np.full(pick.size, p.amp))
    if not tok:
        return np.zeros(0, np.int64), np.zeros(0)
    return np.concatenate(tok).astype(np.int64), np.concatenate(amp)


def mean_query_directions(wl: Workload, q_bits: np.ndarray) -> np.ndarray:
    """Unit mean query direction per (sequence, KV head): float64 [B, Hkv, D]."""
    cuq = wl.cu_qlens()
    g = wl.num_q_heads // wl.num_kv_heads
    q = bf16_bits_to_f32(q_bits).astype(np.float64)
    u = np.zeros((wl.num_seqs, wl.num_kv_heads, wl.head_dim))
    for s in range(wl.num_seqs):
        for kv in range(wl.num_kv_heads):
            m = q[cuq[s]:cuq[s + 1], kv * g:(kv + 1) * g, :].reshape(-1, wl.head_dim).mean(axis=0)
            nrm = np.linalg.norm(m)
            u[s, kv] = m / nrm if nrm > 0 else 0.0
    return u


def plant_patch(wl: Workload, layer: int, q_bits: np.ndarray):
    """Rows of K at ``layer`` that the plants overwrite: (token idx, uint16 [n, Hkv, D]).

    Planted key = bf16(base key + amp * sqrt(D) * u), u the unit mean query
    direction of the key's head group in its sequence."""
    tok, amp = planted_tokens(wl)
    if tok.size == 0:
        return tok, np.zeros((0, wl.num_kv_heads, wl.head_dim), np.uint16)
    u = mean_query_directions(wl, q_bits)
    seq_of = np.searchsorted(wl.cu_seqlens(), tok, side="right") - 1
    row = wl.num_kv_heads * wl.head_dim
    idx = (tok[:, None] * row + np.arange(row)[None, :]).ravel()
    base = bf16_bits_to_f32(normal_bf16_at(wl.seed, TID_K + layer, idx)).astype(np.float64)
    base = base.reshape(tok.size, wl.num_kv_heads, wl.head_dim)
    shifted = base + (amp * np.sqrt(wl.head_dim))[:, None, None] * u[seq_of]
    return tok, f32_to_bf16_bits(shifted.astype(np.float32)).reshape(tok.size, wl.num_kv_heads, wl.head_dim)


def key_slab(wl: Workload, layer: int, q_bits: np.ndarray = None) -> np.ndarray:
    """K of ``layer`` with plants: uint16 [T, Hkv, D]."""
    T = wl.total_tokens
    k = normal_bf16_bits(wl.seed, TID_K + layer, 0, T * wl.num_kv_heads * wl.head_dim)
    k = k.reshape(T, wl.num_kv_heads, wl.head_dim)
    if q_bits is None:
        q_bits = query_rows(wl, layer)
    tok, rows = plant_patch(wl, layer, q_bits)
    k[tok] = rows
    return k


def value_slab(wl: Workload, layer: int) -> np.ndarray:
    T = wl.total_tokens
    return normal_bf16_bits(wl.seed, TID_V + layer, 0, T * wl.num_kv_heads * wl.head_dim).reshape(
        T, wl.num_kv_heads, wl.head_dim)


def plain_key_slab(wl: Workload, layer: int) -> np.ndarray:
    T = wl.total_tokens
    return normal_bf16_bits(wl.seed, TID_K + layer, 0, T * wl.num_kv_heads * wl.head_dim).reshape(
        T, wl.num_kv_heads, wl.head_dim)


def hidden_states(wl: Workload) -> np.ndarray:
    T = wl.total_tokens
    return normal_bf16_bits(wl.seed, TID_HIDDEN, 0, T * wl.hidden).reshape(T, wl.hidden)


def positions(wl: Workload) -> np.ndarray:
    """Per-token metadata row of four int32 (stand-in for multimodal position
    ids): uint32 [T, 4] of hashed bits, so that a wrong row shows."""
    T = wl.total_tokens
    return uniform_u32(wl.seed, TID_POS, np.arange(4 * T, dtype=np.uint64)).reshape(T, 4)


def base_counts(wl: Workload):
    return [(s.n_audio, s.n_visual) for s in wl.seqs]
