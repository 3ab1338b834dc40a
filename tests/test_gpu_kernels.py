"""Kernel-level parity of the CUDA path against the oracle, through the C ABI.

Sizes span several tiles and ragged tails: 256-key blocks and 128-key tiles
of the scoring passes, 126-row (7 heads x 18 tokens) query tiles, 8-CTA
clusters of the selection, 512-byte pieces of the gather.
"""

import numpy as np
import pytest
import torch

import oracle
from parity import check_scores, check_keep
from synth.gen import f32_to_bf16_bits

pytestmark = pytest.mark.gpu

D = 128


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).cuda()


def aligned_ws(ap, seqs):
    n = ap.apack_workspace_size(seqs)
    t = torch.zeros(n + 256, dtype=torch.uint8, device="cuda")
    off = (-t.data_ptr()) % 256
    return t[off:off + n]


def bf16(x):
    return f32_to_bf16_bits(np.asarray(x, np.float32))


def random_batch(rng, lens, nqs, hq, hkv, p_other=0.05, scale_k=1.0, scale_q=1.0):
    mods = []
    for L in lens:
        m = rng.choice([1, 2], L, p=[0.2, 0.8]).astype(np.uint8)
        m[rng.random(L) < p_other] = 0
        mods.append(m)
    mod = np.concatenate(mods) if mods else np.zeros(0, np.uint8)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cuq = np.concatenate([[0], np.cumsum(nqs)]).astype(np.int32)
    T, NQ = int(cu[-1]), int(cuq[-1])
    k = bf16(rng.standard_normal((T, hkv, D)) * scale_k)
    q = bf16(rng.standard_normal((max(NQ, 1), hq, D)) * scale_q)[:NQ]
    na = [int((mod[cu[s]:cu[s + 1]] == 1).sum()) for s in range(len(lens))]
    nv = [int((mod[cu[s]:cu[s + 1]] == 2).sum()) for s in range(len(lens))]
    return mod, cu, cuq, k, q, na, nv


def gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv, softmax_domain=0, q_start=None):
    mod_d = dev(mod)
    seqs = ap.Seqs(cu, cuq, na, nv, mod_d, hq, hkv, softmax_domain=softmax_domain, q_start=q_start)
    ws = aligned_ws(ap, seqs)
    T = int(cu[-1])
    scores = torch.full((max(T, 1),), float("nan"), dtype=torch.float32, device="cuda")
    q_d = dev(q) if q.size else torch.zeros(16, dtype=torch.int16, device="cuda")
    ap.apack_score(seqs, q_d, dev(k), hkv * D * 2, scores, ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    return scores[:T].cpu().numpy()


SHAPES = [
    # lens, n_q per seq, Hq, Hkv
    ([1000], [32], 28, 4),                  # one sequence, 4 key blocks + tail, two query tiles
    ([300, 77, 1290], [5, 1, 40], 28, 4),   # ragged batch, last-query-only sequence
    ([700], [64], 16, 2),                   # 3B heads: 8 per group, exact 128/256-row tiles
    ([513], [3], 4, 4),                     # MHA (group 1)
    ([129, 257, 1], [7, 19, 2], 12, 2),     # tails of one key past a tile
    ([0, 40, 60], [2, 0, 3], 28, 4),        # empty sequence and a sequence without query rows
    ([0, 40, 600], [2, 0, 30], 28, 4),      # the same on the tensor-core path (210 rows per group)
]

# At most 32 query rows per KV head group take the K-read-bound CUDA-core path
# (the paper scores with the last query token only: G = 7 rows per group).
NARROW_SHAPES = [
    ([1000], [1], 28, 4),
    # at most 8 rows per KV head group with 2 or 4 KV heads: the warp-cooperative logits kernel
    ([3000, 700, 1, 0, 90, 64, 65], [1, 1, 1, 1, 0, 1, 1], 28, 4),
    ([5000, 333], [1, 1], 16, 2),           # 3B heads, 8 rows per group
    ([4100], [2], 8, 4),                    # two query tokens, 4 rows per group
    ([777, 1500], [2, 2], 8, 2),            # two query tokens, 8 rows per group
    ([140000], [1], 28, 4),                 # the paper's query row over a 140k-token sequence (8 tiles per CTA)
    # more rows per group: the general logits kernel
    ([3000, 700, 1, 0, 90], [1, 4, 2, 1, 0], 28, 4),
    ([5000], [2], 16, 2),                   # 16 rows per group
    ([2049], [4], 8, 1),                    # 32 rows in one group
]


@pytest.mark.parametrize("lens,nqs,hq,hkv", NARROW_SHAPES)
def test_narrow_path_scores_match_oracle(ap, lens, nqs, hq, hkv):
    rng = np.random.default_rng(sum(lens) * 3 + hq)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, hq, hkv, scale_k=1.5)
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, hq, hkv)
    check_scores(got, ref, strict_rel=2e-3)
    again = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv)
    assert got.tobytes() == again.tobytes()


@pytest.mark.parametrize("lens,nqs,hq,hkv", SHAPES)
def test_scores_match_oracle(ap, lens, nqs, hq, hkv):
    rng = np.random.default_rng(sum(lens) + hq)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, hq, hkv)
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, hq, hkv)
    check_scores(got, ref, strict_rel=2e-3)
    for s in range(len(lens)):      # closed form: scores of a sequence sum to 1 when it has S and queries
        S = ((mod[cu[s]:cu[s + 1]] == 1) | (mod[cu[s]:cu[s + 1]] == 2)).sum()
        tot = got[cu[s]:cu[s + 1]].astype(np.float64).sum()
        assert tot == pytest.approx(1.0 if S and nqs[s] else 0.0, abs=1e-4)


# ------------------------------------------------------------------------------ causal-row domain

CAUSAL_SHAPES = [
    # tensor-core passes (more than 32 rows per head group)
    ([1000], [32], 28, 4),
    ([300, 77, 1290], [5, 1, 40], 28, 4),
    ([700], [64], 16, 2),
    ([513], [40], 4, 4),
    ([129, 257, 40], [7, 19, 2], 12, 2),
    ([40, 600], [0, 30], 28, 4),
    # narrow path: tensor-core logits (<= 8 rows per group, Hkv 2 / 4) and the general kernel
    ([1000], [1], 28, 4),
    ([3000, 700, 1, 90, 64, 65], [1, 1, 1, 0, 1, 1], 28, 4),
    ([5000, 333], [1, 1], 16, 2),
    ([4100], [2], 8, 4),
    ([3000, 700, 2, 90], [1, 4, 2, 0], 28, 4),
    ([2049], [4], 8, 1),
]


@pytest.mark.parametrize("query_text", [False, True])
@pytest.mark.parametrize("lens,nqs,hq,hkv", CAUSAL_SHAPES)
def test_causal_row_scores_match_oracle(ap, lens, nqs, hq, hkv, query_text):
    """APACK_SOFTMAX_CAUSAL_ROW: the denominator is the query token's causal row (every
    token up to the row's position).  query_text: the last n_q tokens (the query rows) are
    text, as in a prompt; otherwise most of them are audio/visual tokens, which then get
    credit only from the rows at or after their position."""
    rng = np.random.default_rng(sum(lens) * 5 + hq + int(query_text))
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, hq, hkv, scale_k=1.3)
    if query_text:
        for s in range(len(lens)):
            mod[cu[s + 1] - nqs[s]:cu[s + 1]] = 0
        na = [int((mod[cu[s]:cu[s + 1]] == 1).sum()) for s in range(len(lens))]
        nv = [int((mod[cu[s]:cu[s + 1]] == 2).sum()) for s in range(len(lens))]
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv, softmax_domain=ap.APACK_SOFTMAX_CAUSAL_ROW)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, hq, hkv, softmax_domain=oracle.SOFTMAX_CAUSAL_ROW)
    check_scores(got, ref, strict_rel=2e-3)
    mm = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv)
    for s in range(len(lens)):      # the causal row spends mass outside S: never more than the S domain's 1
        if nqs[s]:
            assert got[cu[s]:cu[s + 1]].astype(np.float64).sum() <= mm[cu[s]:cu[s + 1]].astype(np.float64).sum() + 1e-4


@pytest.mark.parametrize("lens,nqs,hq,hkv", [CAUSAL_SHAPES[i] for i in (0, 1, 4, 6, 7, 10)])
def test_causal_row_scores_with_the_query_span_inside_the_sequence(ap, lens, nqs, hq, hkv):
    """apack_seqs.q_start_h places each sequence's query rows at a chosen position (text query
    followed by more tokens): row r sees the tokens up to q_start + r, later tokens get nothing
    from any row.  Both scoring paths (tensor-core passes and the few-row path)."""
    rng = np.random.default_rng(sum(lens) * 7 + hq)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, hq, hkv, scale_k=1.3)
    q_start = np.array([int(rng.integers(0, L - n + 1)) for L, n in zip(lens, nqs)], np.int32)
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, hq, hkv, softmax_domain=ap.APACK_SOFTMAX_CAUSAL_ROW,
                     q_start=q_start)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, hq, hkv, softmax_domain=oracle.SOFTMAX_CAUSAL_ROW,
                                  q_start=q_start)
    check_scores(got, ref)
    for s in range(len(lens)):
        if nqs[s]:
            assert not got[cu[s] + q_start[s] + nqs[s]:cu[s + 1]].any()
    # a span that does not fit its sequence is refused before any device work
    bad = q_start.copy()
    bad[-1] = lens[-1] - nqs[-1] + 1
    seqs = ap.Seqs(cu, cuq, na, nv, dev(mod), hq, hkv, softmax_domain=ap.APACK_SOFTMAX_CAUSAL_ROW, q_start=bad)
    with pytest.raises(ap.ApackError) as e:
        ap.apack_workspace_size(seqs)
    assert e.value.status == ap.APACK_EINVAL


def test_select_from_keep_ratios_equals_select_from_counts(ap):
    """apack_select takes the keep ratios of Eq. inner directly (keep_count_h NULL): the same
    kept indices as with the counts apack_keep_counts derives from those ratios."""
    rng = np.random.default_rng(123)
    lens = [3000, 700, 5000]
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, [3, 2, 5], 28, 4)
    scores = rng.random(int(cu[-1])).astype(np.float32)
    scores[(mod != 1) & (mod != 2)] = 0
    mod_d = dev(mod)
    seqs = ap.Seqs(cu, cuq, na, nv, mod_d, 28, 4)
    ratios = np.array([[0.5, 0.25], [0.7, 0.4], [0.33, 0.123]], np.float32)
    counts, new_cu = ap.apack_keep_counts(seqs, ratios)
    ws = aligned_ws(ap, seqs)
    out = []
    for kc, kr in ((counts, None), (None, ratios)):
        keep = torch.full((int(new_cu[-1]),), -1, dtype=torch.int32, device="cuda")
        ap.apack_select(seqs, dev(scores), kc, keep, ws, keep_ratio=kr)
        torch.cuda.synchronize()
        out.append(keep.cpu().numpy())
    np.testing.assert_array_equal(out[0], out[1])
    np.testing.assert_array_equal(out[0], oracle.select_keep(scores, mod, cu, [tuple(c) for c in counts]))
    with pytest.raises(ap.ApackError):
        ap.apack_select(seqs, dev(scores), None, keep, ws, keep_ratio=np.full((3, 2), 1.5, np.float32))


def test_causal_row_domain_rejects_more_rows_than_tokens(ap):
    mod = np.full(10, 1, np.uint8)
    seqs = ap.Seqs(np.array([0, 10], np.int32), np.array([0, 11], np.int32), [10], [0], dev(mod), 28, 4,
                   softmax_domain=ap.APACK_SOFTMAX_CAUSAL_ROW)
    with pytest.raises(ap.ApackError):
        ap.apack_workspace_size(seqs)


def test_scores_large_logits_and_sequence_without_S(ap):
    rng = np.random.default_rng(11)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, [900, 50], [9, 4], 28, 4, scale_k=3.0, scale_q=3.0)
    mod[900:] = 0
    nv[1] = na[1] = 0
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 28, 4)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, 28, 4)
    check_scores(got, ref)
    assert np.all(got[900:] == 0)


@pytest.mark.parametrize("domain", [0, 1])
def test_scores_with_a_logit_far_above_its_run_reference(ap, domain):
    """A late key aligned with one query row gives that row a logit about 190 binary orders of
    magnitude above the maximum of the first key block: the row's online sum would overflow
    its run's fixed reference, so the pass-1 partial is marked and the merge recomputes the
    row's normaliser exactly.  Scores must still match the oracle on every token of S."""
    rng = np.random.default_rng(99 + domain)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, [2000], [5], 28, 4, scale_k=0.05)
    h, r = 9, 2                                    # query head 9 (KV head 1), query row 2
    qv = oracle.bf16_to_f64(q[r, h])
    kv = bf16(12.0 * qv)
    for key in (1500, 1777):
        mod[key] = 2
        k[key, h // 7] = kv
    na = [int((mod == 1).sum())]
    nv = [int((mod == 2).sum())]
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 28, 4, softmax_domain=domain)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, 28, 4, softmax_domain=domain)
    check_scores(got, ref)
    assert ref[1500] > 1e-3 and ref[1777] > 1e-3


def test_scores_identical_keys_are_uniform(ap):
    mod = np.array([0] * 16 + [1, 2, 2, 2] * 300 + [0] * 8, np.uint8)
    T = mod.size
    rng = np.random.default_rng(3)
    k = np.repeat(bf16(rng.standard_normal((1, 4, D))), T, axis=0)
    q = bf16(rng.standard_normal((8, 28, D)))
    got = gpu_scores(ap, mod, np.array([0, T]), np.array([0, 8]), k, q, [300], [900], 28, 4)
    np.testing.assert_allclose(got[mod != 0], 1.0 / 1200, rtol=2e-5)


def test_scores_are_deterministic(ap):
    rng = np.random.default_rng(5)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, [5000, 3000], [64, 17], 28, 4)
    a = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 28, 4)
    b = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 28, 4)
    assert a.tobytes() == b.tobytes()


# ------------------------------------------------------------------------------ selection

def gpu_select(ap, scores, mod, cu, counts, na, nv, mode):
    mod_d = dev(mod)
    seqs = ap.Seqs(cu, np.zeros(len(cu), np.int32), na, nv, mod_d, 28, 4)
    ws = aligned_ws(ap, seqs)
    T = int(cu[-1])
    other = np.diff(cu) - np.asarray(na) - np.asarray(nv)
    counts = np.asarray(counts, np.int32).reshape(-1, 2)
    n_out = int((other + counts[:, 0] + counts[:, 1]).sum())
    keep = torch.full((max(n_out, 1),), -7, dtype=torch.int32, device="cuda")
    mod_o = torch.zeros(max(n_out, 1), dtype=torch.uint8, device="cuda")
    d2s = torch.full((max(T, 1),), -7, dtype=torch.int32, device="cuda")
    ncu = torch.zeros(len(cu), dtype=torch.int32, device="cuda")
    ap.apack_select(seqs, dev(scores.astype(np.float32)), counts, keep, ws, select_mode=mode, modality_out=mod_o,
                    dst_of_src=d2s, new_cu_seqlens=ncu)
    torch.cuda.synchronize()
    err = ap.apack_device_error(ws)
    return (keep[:n_out].cpu().numpy(), mod_o[:n_out].cpu().numpy(), d2s[:T].cpu().numpy(), ncu.cpu().numpy(),
            err)


SEL_CASES = [
    ([2000], "random"), ([1298], "ties"), ([50000, 30, 7000, 0, 1], "random"),
    ([20000], "allequal"), ([100000], "coarse"), ([3, 5, 7, 9, 11, 13, 15, 17, 19, 21] * 7, "coarse"),
    ([400000], "coarse"),   # slices beyond the shared-memory cache: passes read global memory
]


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("lens,kind", SEL_CASES)
def test_select_matches_oracle_exactly(ap, lens, kind, mode):
    rng = np.random.default_rng(len(lens) * 7 + sum(lens) + mode)
    mods = [rng.choice([0, 1, 2], L, p=[0.05, 0.2, 0.75]).astype(np.uint8) for L in lens]
    mod = np.concatenate(mods)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = mod.size
    if kind == "random":
        sc = rng.random(T).astype(np.float32) * 1e-3
    elif kind == "ties":
        sc = (rng.integers(0, 20, T) / 64.0).astype(np.float32)
    elif kind == "coarse":
        sc = (rng.integers(0, 3000, T) * 1e-7).astype(np.float32)
    else:
        sc = np.full(T, 1.0 / 3.0, np.float32)
    sc[(mod != 1) & (mod != 2)] = 0
    na = [int((m == 1).sum()) for m in mods]
    nv = [int((m == 2).sum()) for m in mods]
    counts = []
    for b, (a, v) in enumerate(zip(na, nv)):      # k = 0, k = n and in between
        if mode == 1:
            n = a + v
            counts.append(([n // 3, 0, n, (2 * n) // 3][b % 4], 0))
        else:
            counts.append(([a // 2, 0, a, (a * 7) // 10][b % 4], [(v * 3) // 10, v, 0, v // 4][b % 4]))
    keep, mod_o, d2s, ncu, err = gpu_select(ap, sc, mod, cu, counts, na, nv, mode)
    assert err == ap.APACK_OK
    ref = oracle.select_keep(sc, mod, cu, counts, joint=(mode == 1))
    np.testing.assert_array_equal(keep, ref)
    np.testing.assert_array_equal(mod_o, mod[ref])
    exp_d2s = np.full(T, -1, np.int32)
    exp_d2s[ref] = np.arange(ref.size)
    np.testing.assert_array_equal(d2s, exp_d2s)
    np.testing.assert_array_equal(ncu, oracle.new_cu_seqlens(ref, cu))


def test_select_reports_count_mismatch_without_faulting(ap):
    rng = np.random.default_rng(2)
    mod = rng.choice([0, 1, 2], 5000).astype(np.uint8)
    cu = np.array([0, 5000], np.int32)
    na, nv = int((mod == 1).sum()), int((mod == 2).sum())
    sc = rng.random(5000).astype(np.float32)
    keep, _, _, _, err = gpu_select(ap, sc, mod, cu, [(10, 10)], [na - 1], [nv + 1], 0)
    assert err == ap.APACK_EDEVICE
    assert np.all(keep >= -7) and np.all(keep < 5000)


# ------------------------------------------------------------------------------ compaction

@pytest.mark.parametrize("row_bytes,planes", [(1024, 3), (512, 2), (7168, 1), (4096, 1), (16, 2), (12, 1),
                                              (1, 1), (272, 2)])
def test_compact_is_bitexact(ap, row_bytes, planes):
    rng = np.random.default_rng(row_bytes)
    T = 3001
    src = rng.integers(0, 256, (planes, T, row_bytes), dtype=np.uint8)
    keep = np.sort(rng.choice(T, 1237, replace=False)).astype(np.int32)
    s = dev(src)
    d = torch.zeros((planes, keep.size, row_bytes), dtype=torch.uint8, device="cuda")
    p = ap.make_plane(s, d, row_bytes, planes, src_plane_stride=T * row_bytes,
                      dst_plane_stride=keep.size * row_bytes)
    ap.apack_compact(dev(keep), keep.size, [p])
    torch.cuda.synchronize()
    np.testing.assert_array_equal(d.cpu().numpy(), src[:, keep, :])


def test_compact_many_groups_and_strided_rows(ap):
    rng = np.random.default_rng(9)
    T = 2000
    keep = np.sort(rng.choice(T, 901, replace=False)).astype(np.int32)
    kd = dev(keep)
    groups, outs, refs = [], [], []
    for g, rb in enumerate([1024, 2048, 512, 48]):
        src = rng.integers(0, 256, (2, T, rb + 64), dtype=np.uint8)   # row stride > row bytes
        s = dev(src)
        d = torch.zeros((2, keep.size, rb), dtype=torch.uint8, device="cuda")
        groups.append(ap.make_plane(s, d, rb, 2, src_plane_stride=T * (rb + 64), dst_plane_stride=keep.size * rb,
                                    src_row_stride=rb + 64))
        outs.append((s, d))
        refs.append(src[:, keep, :rb])
    ap.apack_compact(kd, keep.size, groups)
    torch.cuda.synchronize()
    for (s, d), r in zip(outs, refs):
        np.testing.assert_array_equal(d.cpu().numpy(), r)


IN_PLACE_CASES = [
    # T, kept, row bytes, planes, which rows are kept
    (3001, 1237, 1024, 3, "random"),
    (3001, 3001, 1024, 2, "all"),             # every row stays where it is
    (5000, 1, 512, 2, "last"),                # one row moves from the end to row 0
    (20000, 7000, 7168, 1, "random"),         # hidden-state rows, 4 per 32 KB slot
    (40000, 30000, 2048, 3, "tail"),          # a few early rows, then the whole tail: long dependency ranges
    (135272, 58772, 1024, 4, "random"),       # the 10-minute 7B step: thousands of items on every CTA
    (10000, 5000, 1024, 2, "even"),           # every other row: waves of 1, 2, 4, ... rows
    (60000, 51000, 1024, 2, "random"),        # keep ratio 0.85: the item-dependency schedule
]


@pytest.mark.parametrize("T,n_keep,row_bytes,planes,pattern", IN_PLACE_CASES)
def test_compact_in_place_is_bitexact(ap, T, n_keep, row_bytes, planes, pattern):
    """src == dst: the first n_keep rows of every plane become the kept rows (oracle
    compact_rows), the rows after them are left as they were."""
    rng = np.random.default_rng(T + row_bytes + planes)
    src = rng.integers(0, 256, (planes, T, row_bytes), dtype=np.uint8)
    if pattern == "all":
        keep = np.arange(T, dtype=np.int32)
    elif pattern == "last":
        keep = np.array([T - 1], np.int32)
    elif pattern == "even":
        keep = np.arange(0, 2 * n_keep, 2, dtype=np.int32)
    elif pattern == "tail":
        head = np.sort(rng.choice(T // 2, n_keep - (T - T // 2), replace=False))
        keep = np.concatenate([head, np.arange(T // 2, T)]).astype(np.int32)
    else:
        keep = np.sort(rng.choice(T, n_keep, replace=False)).astype(np.int32)
    assert keep.size == n_keep
    buf = dev(src)
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    p = ap.make_plane(buf, buf, row_bytes, planes, src_plane_stride=T * row_bytes, dst_plane_stride=T * row_bytes)
    ap.apack_compact(dev(keep), n_keep, [p], ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    got = buf.cpu().numpy()
    for pl in range(planes):
        np.testing.assert_array_equal(got[pl, :n_keep], oracle.compact_rows(src[pl], keep))
        np.testing.assert_array_equal(got[pl, n_keep:], src[pl, n_keep:])
    # twice in a row on the same workspace: the progress words start from zero again
    buf2 = dev(src)
    p2 = ap.make_plane(buf2, buf2, row_bytes, planes, src_plane_stride=T * row_bytes,
                       dst_plane_stride=T * row_bytes)
    ap.apack_compact(dev(keep), n_keep, [p2], ws=ws)
    torch.cuda.synchronize()
    assert torch.equal(buf2, buf)


def test_compact_in_place_mixed_with_out_of_place_groups(ap):
    rng = np.random.default_rng(31)
    T, rb = 9000, 1024
    keep = np.sort(rng.choice(T, 4100, replace=False)).astype(np.int32)
    a = rng.integers(0, 256, (2, T, rb), dtype=np.uint8)
    b = rng.integers(0, 256, (T, 3584 * 2), dtype=np.uint8)
    ad, bd = dev(a), dev(b)
    bo = torch.zeros((keep.size, 3584 * 2), dtype=torch.uint8, device="cuda")
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    groups = [ap.make_plane(ad, ad, rb, 2, src_plane_stride=T * rb, dst_plane_stride=T * rb),
              ap.make_plane(bd, bo, 3584 * 2, 1)]
    ap.apack_compact(dev(keep), keep.size, groups, ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    np.testing.assert_array_equal(ad.cpu().numpy()[:, :keep.size], a[:, keep])
    np.testing.assert_array_equal(bo.cpu().numpy(), b[keep])


@pytest.mark.parametrize("density", [0.05, 0.43, 0.97])
def test_compact_in_place_several_groups(ap, density):
    """Three in-place groups in one launch (K/V-like 1024 B rows, hidden-like 7168 B rows, 16 B
    metadata rows): every CTA's items run through group boundaries, where the dependency bounds
    restart."""
    rng = np.random.default_rng(int(density * 100))
    T = 30011
    n_keep = max(1, int(T * density))
    keep = np.sort(rng.choice(T, n_keep, replace=False)).astype(np.int32)
    shapes = [(6, 1024), (1, 7168), (1, 16)]
    srcs = [rng.integers(0, 256, (pl, T, rb), dtype=np.uint8) for pl, rb in shapes]
    bufs = [dev(s) for s in srcs]
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    groups = [ap.make_plane(b, b, rb, pl, src_plane_stride=T * rb, dst_plane_stride=T * rb)
              for b, (pl, rb) in zip(bufs, shapes)]
    ap.apack_compact(dev(keep), n_keep, groups, ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    for b, s in zip(bufs, srcs):
        got = b.cpu().numpy()
        for pl in range(s.shape[0]):
            np.testing.assert_array_equal(got[pl, :n_keep], oracle.compact_rows(s[pl], keep))
            np.testing.assert_array_equal(got[pl, n_keep:], s[pl, n_keep:])


def test_compact_in_place_argument_checks(ap):
    T = 100
    keep = dev(np.arange(0, T, 2, dtype=np.int32))
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    buf = torch.zeros((2, T, 40), dtype=torch.uint8, device="cuda")
    with pytest.raises(ap.ApackError):      # rows that are not 16-byte multiples
        ap.apack_compact(keep, T // 2, [ap.make_plane(buf, buf, 40, 2, T * 40, T * 40)], ws=ws)
    buf = torch.zeros((2, T, 64), dtype=torch.uint8, device="cuda")
    with pytest.raises(ap.ApackError):      # no workspace for the progress words
        ap.apack_compact(keep, T // 2, [ap.make_plane(buf, buf, 64, 2, T * 64, T * 64)])
    with pytest.raises(ap.ApackError):      # different layouts on the two sides of one buffer
        ap.apack_compact(keep, T // 2, [ap.make_plane(buf, buf, 64, 2, T * 64, (T // 2) * 64)], ws=ws)


def test_prune_step_in_place_equals_out_of_place(ap):
    rng = np.random.default_rng(44)
    hq, hkv, L, layer, H = 28, 4, 6, 2, 3584
    lens, nqs = [3000, 1500], [40, 3]
    mod, cu, cuq, k0, q, na, nv = random_batch(rng, lens, nqs, hq, hkv)
    T = int(cu[-1])
    nl = L - layer
    row = hkv * D
    kc = torch.from_numpy(rng.integers(-30000, 30000, (nl, T, row), dtype=np.int16)).cuda()
    kc[0] = dev(k0).view(T, row)
    vc = torch.from_numpy(rng.integers(-30000, 30000, (nl, T, row), dtype=np.int16)).cuda()
    hid = torch.from_numpy(rng.integers(-30000, 30000, (T, H), dtype=np.int16)).cuda()
    counts = np.array([[na[0] // 2, nv[0] // 3], [na[1] // 4, nv[1] // 2]], np.int32)
    mod_d = dev(mod)
    seqs = ap.Seqs(cu, cuq, na, nv, mod_d, hq, hkv)
    ws = aligned_ws(ap, seqs)
    n_out = int(T - sum(na) - sum(nv) + counts.sum())

    def outs():
        return (torch.empty(max(n_out, 1), dtype=torch.int32, device="cuda"),
                torch.empty(max(n_out, 1), dtype=torch.uint8, device="cuda"),
                torch.empty(T, dtype=torch.float32, device="cuda"))

    keep1, mo1, sc1 = outs()
    ko = torch.empty((nl, n_out, row), dtype=torch.int16, device="cuda")
    vo = torch.empty_like(ko)
    ho = torch.empty((n_out, H), dtype=torch.int16, device="cuda")
    cu1 = ap.apack_prune_step(seqs, layer, L, dev(q), kc, vc, T * row * 2, hid, H, keep_count=counts,
                              k_out=ko, v_out=vo, kv_out_layer_stride=n_out * row * 2, hidden_out=ho,
                              modality_out=mo1, keep_idx=keep1, scores=sc1, ws=ws)
    keep2, mo2, sc2 = outs()
    kc2, vc2, hid2 = kc.clone(), vc.clone(), hid.clone()
    cu2 = ap.apack_prune_step(seqs, layer, L, dev(q), kc2, vc2, T * row * 2, hid2, H, keep_count=counts,
                              k_out=kc2, v_out=vc2, kv_out_layer_stride=T * row * 2, hidden_out=hid2,
                              modality_out=mo2, keep_idx=keep2, scores=sc2, ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    np.testing.assert_array_equal(cu1, cu2)
    assert torch.equal(keep1[:n_out], keep2[:n_out]) and torch.equal(mo1[:n_out], mo2[:n_out])
    assert torch.equal(kc2[:, :n_out], ko) and torch.equal(vc2[:, :n_out], vo) and torch.equal(hid2[:n_out], ho)
    with pytest.raises(ap.ApackError):      # in place needs both caches in place, at the input's slab stride
        ap.apack_prune_step(seqs, layer, L, dev(q), kc2, vc2, T * row * 2, hid2, H, keep_count=counts,
                            k_out=kc2, v_out=vo, kv_out_layer_stride=T * row * 2, hidden_out=hid2,
                            modality_out=mo2, keep_idx=keep2, scores=sc2, ws=ws)


@pytest.mark.parametrize("row_bytes,planes", [(1024, 3), (7168, 1), (48, 2)])
def test_compact_from_pinned_host_memory(ap, row_bytes, planes):
    """A group whose source is pinned host memory is gathered over the host link (zero
    copy): only kept rows are read; the result is the same bytes as from device memory."""
    rng = np.random.default_rng(row_bytes + 5)
    T = 20011
    src = rng.integers(0, 256, (planes, T, row_bytes), dtype=np.uint8)
    keep = np.sort(rng.choice(T, 8123, replace=False)).astype(np.int32)
    h = torch.from_numpy(src).pin_memory()
    d = torch.zeros((planes, keep.size, row_bytes), dtype=torch.uint8, device="cuda")
    p = ap.make_plane(h, d, row_bytes, planes, src_plane_stride=T * row_bytes, dst_plane_stride=keep.size * row_bytes)
    ap.apack_compact(dev(keep), keep.size, [p])
    torch.cuda.synchronize()
    got = d.cpu().numpy()
    for pl in range(planes):
        np.testing.assert_array_equal(got[pl], oracle.compact_rows(src[pl], keep))


def test_host_memory_is_refused_where_tma_reads_it(ap):
    rng = np.random.default_rng(3)
    mod, cu, cuq, k, q, na, nv = random_batch(rng, [300], [4], 28, 4)
    seqs = ap.Seqs(cu, cuq, na, nv, dev(mod), 28, 4)
    ws = aligned_ws(ap, seqs)
    scores = torch.zeros(300, dtype=torch.float32, device="cuda")
    k_host = torch.from_numpy(k.view(np.int16)).pin_memory()
    with pytest.raises(ap.ApackError) as e:
        ap.apack_score(seqs, dev(q), k_host, 4 * D * 2, scores, ws)
    assert e.value.status == ap.APACK_EINVAL
    h = torch.zeros((2, 64, 64), dtype=torch.uint8).pin_memory()
    with pytest.raises(ap.ApackError) as e:      # a host buffer cannot be compacted in place
        ap.apack_compact(dev(np.arange(0, 64, 2, dtype=np.int32)), 32, [ap.make_plane(h, h, 64, 2, 4096, 4096)],
                         ws=ws)
    assert e.value.status == ap.APACK_EINVAL


def test_device_fill_matches_host_generator(ap):
    from synth.device import fill_normal_bf16
    from synth.gen import normal_bf16_bits
    t = torch.empty(1 << 20, dtype=torch.int16, device="cuda")
    fill_normal_bf16(t, 3, 2004, start=12345)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(t.cpu().numpy().view(np.uint16), normal_bf16_bits(3, 2004, 12345, 1 << 20))


def test_compact_strided_destination_rows(ap):
    # output rows with a larger stride than the row: the copy stores row by row
    rng = np.random.default_rng(10)
    T, rb, pad = 1500, 1024, 512
    keep = np.sort(rng.choice(T, 700, replace=False)).astype(np.int32)
    src = rng.integers(0, 256, (3, T, rb), dtype=np.uint8)
    s = dev(src)
    d = torch.zeros((3, keep.size, rb + pad), dtype=torch.uint8, device="cuda")
    p = ap.make_plane(s, d, rb, 3, src_plane_stride=T * rb, dst_plane_stride=keep.size * (rb + pad),
                      dst_row_stride=rb + pad)
    ap.apack_compact(dev(keep), keep.size, [p])
    torch.cuda.synchronize()
    out = d.cpu().numpy()
    np.testing.assert_array_equal(out[:, :, :rb], src[:, keep, :])
    assert not out[:, :, rb:].any()


# ------------------------------------------------------------------------------ batch limits

@pytest.mark.parametrize("path", ["narrow", "wide"])
def test_scores_batch_beyond_one_launch(ap, path):
    # 70 sequences: more than one launch's 64, on both scoring paths
    rng = np.random.default_rng(70 if path == "narrow" else 71)
    lens = [int(x) for x in rng.integers(0, 400, 70)]
    nqs = [int(x) for x in (rng.integers(0, 4, 70) if path == "narrow" else rng.integers(5, 41, 70))]
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, 28, 4)
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 28, 4)
    check_scores(got, oracle.relevance_scores(q, k, cu, cuq, mod, 28, 4))


def test_maximum_number_of_sequences(ap):
    # APACK_MAX_SEQS short sequences through scoring (narrow path) and selection
    rng = np.random.default_rng(4096)
    B = 4096
    lens = [int(x) for x in rng.integers(0, 40, B)]
    nqs = [int(x) for x in rng.integers(0, 2, B)]
    mod, cu, cuq, k, q, na, nv = random_batch(rng, lens, nqs, 4, 2)
    got = gpu_scores(ap, mod, cu, cuq, k, q, na, nv, 4, 2)
    ref = oracle.relevance_scores(q, k, cu, cuq, mod, 4, 2)
    check_scores(got, ref)
    counts = [(a // 2, (v * 3) // 4) for a, v in zip(na, nv)]
    keep, mod_o, _, ncu, err = gpu_select(ap, got, mod, cu, counts, na, nv, 0)
    assert err == ap.APACK_OK
    ref_keep = oracle.select_keep(got, mod, cu, counts)
    np.testing.assert_array_equal(keep, ref_keep)
    np.testing.assert_array_equal(ncu, oracle.new_cu_seqlens(ref_keep, cu))
