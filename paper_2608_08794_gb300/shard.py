"""Splitting a packed batch across GPUs by whole sequences.

The prune step of Sec. 3.2 works on each sequence alone: its scores, its
top-k and its compaction never read another sequence's tokens.  So a ragged
batch spreads over several GPUs (one process per GPU) by giving each rank a
set of whole sequences.  No exchange is needed on the data path: every rank
keeps the compacted caches of its own sequences.

This module is host-side bookkeeping only (which rank runs which sequence,
and the index maps between a rank's packed sub-batch and the whole batch);
the step itself runs in the library on each rank.

* ``plan_by_sequence`` balances the ranks by token count (longest sequence
  first onto the least-loaded rank), then lists each rank's sequences in their
  original order.
* ``SequenceShard`` packs one rank's sequences into a contiguous sub-batch
  (its own ``cu_seqlens`` / ``cu_qlens``, counts and keep counts) and maps the
  sub-batch's token and query rows back to the whole batch's.
* ``merge_keep`` / ``merge_cu_seqlens`` assemble the whole batch's kept
  indices and new offsets from every rank's results (verification and
  reporting only; the step does not need them).
"""

import numpy as np


def plan_by_sequence(cu_seqlens, world, weights=None):
    """Sequence ids per rank, balanced by tokens (or by `weights` per sequence).

    Greedy longest-processing-time assignment: sequences in decreasing weight
    (ties: lower id first) each go to the rank with the least weight so far
    (ties: lower rank).  Each rank's list is returned in ascending id order, so
    that its sub-batch keeps the batch's sequence order.  A rank may get no
    sequence when there are fewer sequences than ranks."""
    cu = np.asarray(cu_seqlens, np.int64)
    n = len(cu) - 1
    if world < 1:
        raise ValueError("world size must be at least 1")
    w = np.diff(cu) if weights is None else np.asarray(weights, np.int64)
    if w.shape != (n,):
        raise ValueError("one weight per sequence")
    order = sorted(range(n), key=lambda b: (-int(w[b]), b))
    load = [0] * world
    out = [[] for _ in range(world)]
    for b in order:
        r = min(range(world), key=lambda x: (load[x], x))
        out[r].append(b)
        load[r] += int(w[b])
    return [np.asarray(sorted(x), np.int64) for x in out]


class SequenceShard:
    """One rank's sequences, packed contiguously.

    seq_ids: ascending sequence ids of the whole batch.  The sub-batch's token
    t of local sequence j is token ``cu_seqlens[seq_ids[j]] + t`` of the batch;
    ``token_index`` / ``q_index`` hold these maps for every local token and
    query row."""

    def __init__(self, seq_ids, cu_seqlens, cu_qlens, n_audio, n_visual):
        ids = np.asarray(seq_ids, np.int64)
        if ids.size and (np.any(np.diff(ids) <= 0) or ids[0] < 0 or ids[-1] >= len(cu_seqlens) - 1):
            raise ValueError("sequence ids must be ascending, distinct and in range")
        cu = np.asarray(cu_seqlens, np.int64)
        cq = np.asarray(cu_qlens, np.int64)
        self.seq_ids = ids
        lens, qlens = cu[ids + 1] - cu[ids], cq[ids + 1] - cq[ids]
        self.cu_seqlens = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
        self.cu_qlens = np.concatenate([[0], np.cumsum(qlens)]).astype(np.int32)
        self.n_audio = np.asarray(n_audio, np.int32)[ids]
        self.n_visual = np.asarray(n_visual, np.int32)[ids]
        self.token_index = np.concatenate([np.arange(cu[b], cu[b + 1]) for b in ids]).astype(np.int64) \
            if ids.size else np.zeros(0, np.int64)
        self.q_index = np.concatenate([np.arange(cq[b], cq[b + 1]) for b in ids]).astype(np.int64) \
            if ids.size else np.zeros(0, np.int64)

    @property
    def num_seqs(self):
        return int(self.seq_ids.size)

    @property
    def total_tokens(self):
        return int(self.cu_seqlens[-1])

    def keep_counts(self, counts):
        """This rank's rows of a whole-batch keep-count array [B, 2]."""
        return np.asarray(counts, np.int32).reshape(-1, 2)[self.seq_ids]

    def tokens(self, per_token):
        """This rank's rows of a whole-batch per-token array (numpy or torch)."""
        idx = self.token_index
        if hasattr(per_token, "index_select"):
            import torch
            return per_token.index_select(0, torch.from_numpy(idx).to(per_token.device))
        return np.asarray(per_token)[idx]

    def query_rows(self, per_row):
        """This rank's rows of the whole batch's packed query rows."""
        idx = self.q_index
        if hasattr(per_row, "index_select"):
            import torch
            return per_row.index_select(0, torch.from_numpy(idx).to(per_row.device))
        return np.asarray(per_row)[idx]

    def to_global(self, local_keep):
        """Whole-batch token indices of a sub-batch's kept indices (ascending stays ascending)."""
        return self.token_index[np.asarray(local_keep, np.int64)]


def merge_keep(global_keeps):
    """The whole batch's kept indices from every rank's (already global) kept indices."""
    parts = [np.asarray(k, np.int64) for k in global_keeps if len(k)]
    if not parts:
        return np.zeros(0, np.int64)
    out = np.sort(np.concatenate(parts))
    if out.size > 1 and np.any(np.diff(out) == 0):
        raise ValueError("two ranks kept the same token: the shards overlap")
    return out


def merge_cu_seqlens(shards, local_new_cu, num_seqs):
    """The whole batch's offsets after the step, from each rank's new local offsets."""
    kept = np.zeros(num_seqs, np.int64)
    seen = np.zeros(num_seqs, bool)
    for sh, cu in zip(shards, local_new_cu):
        cu = np.asarray(cu, np.int64)
        if cu.size != sh.num_seqs + 1:
            raise ValueError("offsets do not match the shard")
        kept[sh.seq_ids] = np.diff(cu)
        seen[sh.seq_ids] = True
    if not seen.all():
        raise ValueError("a sequence belongs to no shard")
    return np.concatenate([[0], np.cumsum(kept)]).astype(np.int32)
