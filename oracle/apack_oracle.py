"""Plain, slow, fp64 CPU oracle of the A-PACK inner-LLM prune step.

TEST INFRASTRUCTURE: this module exists to check the CUDA library.  Only
``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` leg of
``bench.py`` may import it.  It shares no code with the CUDA path.

What the step computes (A-PACK, Sec. 3.2 "Inner-LLM Query-Aware
Compression", Eq. (inner_score) and Eq. (inner); Algorithm 1, the inner-LLM
loop; Table S-hparams "Query score"):

1. Relevance (Eq. inner_score).  For a sequence with cached multimodal token
   set S (audio and visual tokens), a query vector q and keys k_i,
   I_i = exp(q.k_i / sqrt(d)) / sum_{j in S} exp(q.k_j / sqrt(d)), i in S,
   with d the key dimension.  For a multi-head decoder the score is averaged
   over attention heads.  Readings taken here: the average runs over all
   query heads h (each with its own query vector) and over every row r of
   the caller's query span (the paper's setting is a span of one row, the
   last query token); query head h reads key head h // (Hq / Hkv)
   (grouped-query attention with contiguous groups); tokens outside S score 0.
2. Selection (Eq. inner).  S <- TopK over ceil((1-P)|S|) tokens by I.  Taken
   here per (sequence, modality) with keep ratio r = 1-P given per modality
   (or jointly over S, the paper's literal form); ties go to the lower token
   index; tokens outside S are always kept; kept tokens stay in their
   original order.
3. Compaction (Sec. 3.2, last sentence; Algorithm 1, "slice their KV-cache
   entries").  Every per-token row of every plane (K and V of the compacted
   layers, hidden states, metadata) is copied so that output row j is input
   row keep_idx[j].

A second softmax domain reads "the full key row" as the decoder's own
attention row: the denominator of Eq. (inner_score) then runs over the
causal attention row of the query token, i.e. every token at or before the
query row's position (system, text, audio, visual and query tokens), with the
query rows at a given position of the sequence (by default its last n_q
tokens); a token of S after a row's position gets nothing from that row.

The arithmetic is fp64 from exactly widened bf16 inputs; numpy's matmul,
exp and stable argsort are the only library steps.
"""

import math

import numpy as np

MOD_OTHER, MOD_AUDIO, MOD_VISUAL = 0, 1, 2
SOFTMAX_MM, SOFTMAX_CAUSAL_ROW = 0, 1


def bf16_to_f64(bits):
    """Exact widening of bf16 bit patterns (uint16) to float64."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def relevance_scores(q_bits, k_bits, cu_seqlens, cu_qlens, modality, num_q_heads, num_kv_heads,
                     row_chunk=512, softmax_domain=SOFTMAX_MM, q_start=None):
    """Eq. (inner_score), averaged over query heads and query rows.

    q_bits: uint16 [sum n_q, Hq, D] (bf16) query rows, packed per sequence by cu_qlens.
    k_bits: uint16 [T, Hkv, D] (bf16) keys of the pruning layer, packed by cu_seqlens.
    modality: uint8 [T]; 1 = audio, 2 = visual form S, anything else is outside S.
    softmax_domain: SOFTMAX_MM (the denominator over S, as Eq. inner_score prints it) or
    SOFTMAX_CAUSAL_ROW (over the causal attention row; see the module docstring).
    q_start: per sequence, the position of its first query row (causal domain only);
    None puts the query rows at the end of each sequence.
    Returns float64 [T]; 0 outside S.
    """
    if softmax_domain == SOFTMAX_CAUSAL_ROW:
        return _relevance_causal(q_bits, k_bits, cu_seqlens, cu_qlens, modality, num_q_heads, num_kv_heads,
                                 q_start)
    q_bits = np.asarray(q_bits)
    k_bits = np.asarray(k_bits)
    T = k_bits.shape[0]
    D = k_bits.shape[2]
    group = num_q_heads // num_kv_heads
    scores = np.zeros(T, dtype=np.float64)
    for s in range(len(cu_seqlens) - 1):
        t0, t1 = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        r0, r1 = int(cu_qlens[s]), int(cu_qlens[s + 1])
        n_q = r1 - r0
        mm = np.nonzero((modality[t0:t1] == MOD_AUDIO) | (modality[t0:t1] == MOD_VISUAL))[0] + t0
        if mm.size == 0 or n_q == 0:
            continue
        acc = np.zeros(mm.size, dtype=np.float64)
        for h in range(num_q_heads):
            g = h // group
            keys = bf16_to_f64(k_bits[mm, g, :])                 # [|S|, D]
            for c0 in range(r0, r1, row_chunk):
                c1 = min(r1, c0 + row_chunk)
                qs = bf16_to_f64(q_bits[c0:c1, h, :])            # [rows, D]
                x = (qs @ keys.T) / math.sqrt(D)                 # logits q.k / sqrt(d)
                x = x - x.max(axis=1, keepdims=True)             # softmax over j in S
                p = np.exp(x)
                p /= p.sum(axis=1, keepdims=True)
                acc += p.sum(axis=0)
        scores[mm] = acc / (num_q_heads * n_q)                   # mean over heads and rows
    return scores


def _relevance_causal(q_bits, k_bits, cu_seqlens, cu_qlens, modality, num_q_heads, num_kv_heads, q_start=None):
    """Eq. (inner_score) with the causal-row denominator: query row r of a
    sequence of length L with n_q query rows is token p_r = q_start + r (q_start =
    L - n_q when not given); its softmax runs over the tokens 0..p_r of the
    sequence, and the score of a token i of S averages that row's probability of
    i (0 when i > p_r) over heads and rows."""
    q_bits = np.asarray(q_bits)
    k_bits = np.asarray(k_bits)
    T = k_bits.shape[0]
    D = k_bits.shape[2]
    group = num_q_heads // num_kv_heads
    scores = np.zeros(T, dtype=np.float64)
    for s in range(len(cu_seqlens) - 1):
        t0, t1 = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        r0, r1 = int(cu_qlens[s]), int(cu_qlens[s + 1])
        n_q, L = r1 - r0, t1 - t0
        in_s = (modality[t0:t1] == MOD_AUDIO) | (modality[t0:t1] == MOD_VISUAL)
        if not in_s.any() or n_q == 0:
            continue
        acc = np.zeros(L, dtype=np.float64)
        for h in range(num_q_heads):
            keys = bf16_to_f64(k_bits[t0:t1, h // group, :])     # [L, D], every token
            for r in range(n_q):
                p = (L - n_q if q_start is None else int(q_start[s])) + r   # position of query row r
                qv = bf16_to_f64(q_bits[r0 + r, h, :])
                x = (keys[:p + 1] @ qv) / math.sqrt(D)            # the row's visible logits
                e = np.exp(x - x.max())
                acc[:p + 1] += e / e.sum()
        scores[t0:t1] = np.where(in_s, acc / (num_q_heads * n_q), 0.0)
    return scores


def keep_count(ratio, n):
    """ceil((1-P) * n) of Eq. (inner) with the keep ratio (1-P) read on a 1e-6
    grid, so that e.g. 0.7 * 3000 gives exactly 2100 (integer arithmetic)."""
    if not (0.0 <= ratio <= 1.0):
        raise ValueError("keep ratio outside [0, 1]")
    num = int(math.floor(ratio * 1e6 + 0.5))
    return min(int(n), -((-num * int(n)) // 1000000))


def step_keep_counts(ratios, base_counts):
    """Keep counts of one step: ratios[s] = (audio, visual) applied to the
    per-sequence counts base_counts[s] = (n_audio, n_visual) (cumulative
    ratios are applied to the counts entering the first step)."""
    return [(keep_count(ra, na), keep_count(rv, nv)) for (ra, rv), (na, nv) in zip(ratios, base_counts)]


def select_keep(scores, modality, cu_seqlens, keep_counts, joint=False):
    """Eq. (inner): per segment, the k highest-scoring tokens; a stable sort of
    -score keeps the lower index first among equal scores.  Tokens outside S
    are kept.  Returns the kept token indices, ascending (original order).

    keep_counts[s] = (k_audio, k_visual), or with joint=True (k_S, unused)
    for one segment over both modalities.
    """
    scores = np.asarray(scores)
    out = []
    for s in range(len(cu_seqlens) - 1):
        t0, t1 = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        idx = np.arange(t0, t1)
        mod = modality[t0:t1]
        keep = [idx[(mod != MOD_AUDIO) & (mod != MOD_VISUAL)]]
        if joint:
            segs = [(((mod == MOD_AUDIO) | (mod == MOD_VISUAL)), keep_counts[s][0])]
        else:
            segs = [(mod == MOD_AUDIO, keep_counts[s][0]), (mod == MOD_VISUAL, keep_counts[s][1])]
        for mask, k in segs:
            cand = idx[mask]
            if k > cand.size:
                raise ValueError("keep count larger than the segment")
            order = np.argsort(-scores[cand], kind="stable")
            keep.append(cand[order[:k]])
        out.append(np.sort(np.concatenate(keep)))
    return np.concatenate(out).astype(np.int64) if out else np.zeros(0, np.int64)


def new_cu_seqlens(keep_idx, cu_seqlens):
    """Packed offsets of the kept tokens per sequence."""
    counts = np.searchsorted(keep_idx, np.asarray(cu_seqlens[1:]), side="left")
    return np.concatenate([[0], counts]).astype(np.int32)


def compact_rows(plane, keep_idx):
    """Sec. 3.2 slicing: output row j is input row keep_idx[j] (a copy)."""
    return np.ascontiguousarray(np.asarray(plane)[np.asarray(keep_idx)])


def prune_step(q_bits, k_bits, cu_seqlens, cu_qlens, modality, num_q_heads, num_kv_heads,
               keep_counts, planes=(), joint=False, softmax_domain=SOFTMAX_MM):
    """One inner-LLM pruning step: scores, kept indices, new offsets and the
    compacted planes (each a per-token array, first axis = token)."""
    scores = relevance_scores(q_bits, k_bits, cu_seqlens, cu_qlens, modality, num_q_heads, num_kv_heads,
                              softmax_domain=softmax_domain)
    keep_idx = select_keep(scores, modality, cu_seqlens, keep_counts, joint=joint)
    return dict(scores=scores, keep_idx=keep_idx,
                cu_seqlens=new_cu_seqlens(keep_idx, cu_seqlens),
                modality=compact_rows(modality, keep_idx),
                planes=[compact_rows(p, keep_idx) for p in planes])


def score_tolerance(ref):
    """The comparison rule for relevance scores: |x - ref| <= 1e-5 + 2e-3 |ref|
    (fp32 accumulation of bf16 inputs against this fp64 oracle)."""
    return 1e-5 + 2e-3 * np.abs(ref)
