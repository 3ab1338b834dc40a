"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

Each test targets a plausible slip in the oracle: a dropped or wrong scale
(1/sqrt(d)), a softmax over the wrong set (including tokens outside S), an
average over the wrong axis, the wrong head grouping, a wrong tie rule, a
wrong rounding of ceil((1-P)|S|), a reordered output.  None of them re-types
the oracle's own formula: they use brute force with a different algorithm
(arbitrary-precision sums and rank counting), closed forms, invariants and
special cases that reduce to library routines.
"""

import math

import mpmath
import numpy as np
import pytest
import scipy.special

import oracle
from synth.gen import f32_to_bf16_bits

pytestmark = pytest.mark.filterwarnings("ignore")

D = 128


def bf16(x):
    return f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def rand_bf16(rng, shape, scale=1.0):
    return bf16(rng.standard_normal(shape) * scale)


def one_seq(modality):
    modality = np.asarray(modality, np.uint8)
    return np.array([0, modality.size], np.int32), modality


def brute_scores(q_bits, k_bits, cu, cuq, mod, Hq, Hkv):
    """Arbitrary-precision reference: explicit double loop, mpmath exp and
    sums at 40 digits, no vectorised softmax."""
    mpmath.mp.dps = 40
    q = oracle.bf16_to_f64(q_bits)
    k = oracle.bf16_to_f64(k_bits)
    T = k.shape[0]
    out = [mpmath.mpf(0)] * T
    g = Hq // Hkv
    for s in range(len(cu) - 1):
        S = [i for i in range(cu[s], cu[s + 1]) if mod[i] in (1, 2)]
        rows = range(cuq[s], cuq[s + 1])
        if not S or not rows:
            continue
        for h in range(Hq):
            for r in rows:
                logits = [mpmath.fsum(mpmath.mpf(float(a)) * mpmath.mpf(float(b))
                                      for a, b in zip(q[r, h], k[i, h // g])) / mpmath.sqrt(D) for i in S]
                z = mpmath.fsum(mpmath.exp(x) for x in logits)
                for i, x in zip(S, logits):
                    out[i] += mpmath.exp(x) / z
        for i in S:
            out[i] /= Hq * len(rows)
    return np.array([float(v) for v in out])


def brute_select(scores, mod, cu, counts, joint=False):
    """Rank counting: token i is kept iff fewer than k tokens of its segment
    beat it (higher score, or equal score and lower index)."""
    kept = []
    for s in range(len(cu) - 1):
        for i in range(cu[s], cu[s + 1]):
            if mod[i] not in (1, 2):
                kept.append(i)
                continue
            seg = (lambda j: mod[j] in (1, 2)) if joint else (lambda j, m=mod[i]: mod[j] == m)
            k = counts[s][0] if (joint or mod[i] == 1) else counts[s][1]
            beat = sum(1 for j in range(cu[s], cu[s + 1]) if seg(j) and
                       (scores[j] > scores[i] or (scores[j] == scores[i] and j < i)))
            if beat < k:
                kept.append(i)
    return np.array(kept, np.int64)


@pytest.mark.parametrize("Hq,Hkv,nq", [(4, 2, 3), (2, 2, 1), (6, 1, 2)])
def test_scores_match_arbitrary_precision_brute_force(Hq, Hkv, nq):
    rng = np.random.default_rng(Hq * 10 + Hkv)
    mod = np.array([0, 0, 1, 2, 2, 1, 2, 2, 2, 1, 0, 2, 1, 1, 0], np.uint8)
    mod2 = np.array([0, 2, 2, 1, 2, 1, 0, 0], np.uint8)
    modality = np.concatenate([mod, mod2])
    cu = np.array([0, mod.size, modality.size], np.int32)
    cuq = np.array([0, nq, 2 * nq], np.int32)
    k = rand_bf16(rng, (modality.size, Hkv, D))
    q = rand_bf16(rng, (2 * nq, Hq, D), 0.3)
    got = oracle.relevance_scores(q, k, cu, cuq, modality, Hq, Hkv)
    ref = brute_scores(q, k, cu, cuq, modality, Hq, Hkv)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-15)


def test_two_token_closed_form_pins_scale_and_sign():
    # q = 8 e0, k1 = 2 e0, k2 = -1 e0 -> q.k = 16, -8; with scale 1/sqrt(128)
    # I_1 = 1 / (1 + exp(-(16 + 8)/sqrt(128))) (a logistic function).
    q = np.zeros((1, 1, D), np.float32); q[0, 0, 0] = 8
    k = np.zeros((3, 1, D), np.float32); k[1, 0, 0] = 2; k[2, 0, 0] = -1; k[0, 0, 0] = 100
    cu, mod = one_seq([0, 1, 2])
    got = oracle.relevance_scores(bf16(q), bf16(k), cu, np.array([0, 1]), mod, 1, 1)
    i1 = 1.0 / (1.0 + math.exp(-24.0 / math.sqrt(128.0)))
    assert got[0] == 0.0
    assert got[1] == pytest.approx(i1, rel=1e-14)
    assert got[2] == pytest.approx(1.0 - i1, rel=1e-13)


def test_tokens_outside_S_do_not_enter_the_denominator():
    rng = np.random.default_rng(1)
    mod = np.array([0, 1, 2, 1, 0, 2, 0], np.uint8)
    k = rand_bf16(rng, (mod.size, 2, D))
    q = rand_bf16(rng, (2, 4, D))
    cu, _ = one_seq(mod)
    a = oracle.relevance_scores(q, k, cu, np.array([0, 2]), mod, 4, 2)
    k2 = k.copy()
    k2[[0, 4, 6]] = bf16(np.full((3, 2, D), 30.0))   # huge logits on non-S tokens
    b = oracle.relevance_scores(q, k2, cu, np.array([0, 2]), mod, 4, 2)
    np.testing.assert_array_equal(a, b)
    assert np.all(a[[0, 4, 6]] == 0)


def test_single_head_single_row_equals_library_softmax():
    rng = np.random.default_rng(2)
    mod = np.full(50, 2, np.uint8); mod[:5] = 0; mod[10:20] = 1
    k = rand_bf16(rng, (50, 1, D))
    q = rand_bf16(rng, (1, 1, D))
    cu, _ = one_seq(mod)
    got = oracle.relevance_scores(q, k, cu, np.array([0, 1]), mod, 1, 1)
    S = np.nonzero(mod != 0)[0]
    kk = oracle.bf16_to_f64(k)[S, 0, :]
    qq = oracle.bf16_to_f64(q)[0, 0, :]
    ref = scipy.special.softmax(kk @ qq / np.sqrt(D))
    np.testing.assert_allclose(got[S], ref, rtol=1e-13)


def test_identical_keys_and_zero_query_give_uniform_scores():
    rng = np.random.default_rng(3)
    mod = np.array([0] * 3 + [1, 2] * 20 + [0] * 2, np.uint8)
    cu, _ = one_seq(mod)
    kk = rand_bf16(rng, (1, 2, D))
    k = np.repeat(kk, mod.size, axis=0)
    q = rand_bf16(rng, (3, 4, D))
    got = oracle.relevance_scores(q, k, cu, np.array([0, 3]), mod, 4, 2)
    S = np.nonzero(mod != 0)[0]
    np.testing.assert_allclose(got[S], 1.0 / S.size, rtol=1e-14)
    qz = np.zeros_like(q)
    got0 = oracle.relevance_scores(qz, rand_bf16(rng, k.shape), cu, np.array([0, 3]), mod, 4, 2)
    np.testing.assert_allclose(got0[S], 1.0 / S.size, rtol=1e-14)


def test_scores_sum_to_one_per_sequence():
    rng = np.random.default_rng(4)
    mod = np.concatenate([np.array([0, 1, 2, 2, 1, 0]), np.array([0] + [2] * 30 + [1] * 9 + [0] * 4)]).astype(np.uint8)
    cu = np.array([0, 6, mod.size], np.int32)
    k = rand_bf16(rng, (mod.size, 4, D), 2.0)
    q = rand_bf16(rng, (5, 28, D))
    got = oracle.relevance_scores(q, k, cu, np.array([0, 1, 5]), mod, 28, 4)
    assert got[:6].sum() == pytest.approx(1.0, abs=1e-13)
    assert got[6:].sum() == pytest.approx(1.0, abs=1e-13)


def test_grouped_query_attention_equals_repeated_kv_heads():
    # query head h reads key head h // (Hq/Hkv): contiguous groups
    rng = np.random.default_rng(5)
    mod = np.array([0] + [1, 2, 2] * 10 + [0], np.uint8)
    cu, _ = one_seq(mod)
    k = rand_bf16(rng, (mod.size, 2, D))
    q = rand_bf16(rng, (2, 6, D))
    gqa = oracle.relevance_scores(q, k, cu, np.array([0, 2]), mod, 6, 2)
    mha = oracle.relevance_scores(q, np.repeat(k, 3, axis=1), cu, np.array([0, 2]), mod, 6, 6)
    np.testing.assert_allclose(gqa, mha, rtol=1e-14, atol=0)
    # interleaved grouping (h % Hkv) gives a different answer on the same data
    inter = oracle.relevance_scores(q, np.tile(k, (1, 3, 1)), cu, np.array([0, 2]), mod, 6, 6)
    assert np.max(np.abs(inter - gqa)) > 1e-6


def test_average_over_query_rows_and_heads():
    # Hq=2 heads, 2 rows: each (head,row) sees a two-token softmax with a
    # known logit gap; the score is the plain mean of the four logistic values.
    q = np.zeros((2, 2, D), np.float32)
    gaps = np.array([[1.0, 2.0], [4.0, -3.0]])        # [row, head] -> q[row,h,0]
    q[:, :, 0] = gaps
    k = np.zeros((2, 1, D), np.float32); k[0, 0, 0] = 1.0   # x1 - x2 = gap / sqrt(128)
    cu, mod = one_seq([1, 2])
    got = oracle.relevance_scores(bf16(q), bf16(k), cu, np.array([0, 2]), mod, 2, 1)
    ref = np.mean(1.0 / (1.0 + np.exp(-gaps / np.sqrt(128.0))))
    assert got[0] == pytest.approx(ref, rel=1e-14)


def test_permutation_within_S_permutes_scores():
    rng = np.random.default_rng(6)
    mod = np.array([0, 0] + [1] * 12 + [2] * 20 + [0], np.uint8)
    cu, _ = one_seq(mod)
    k = rand_bf16(rng, (mod.size, 2, D))
    q = rand_bf16(rng, (2, 4, D))
    a = oracle.relevance_scores(q, k, cu, np.array([0, 2]), mod, 4, 2)
    perm = np.arange(mod.size)
    perm[2:34] = 2 + rng.permutation(32)
    b = oracle.relevance_scores(q, k[perm], cu, np.array([0, 2]), mod[perm], 4, 2)
    np.testing.assert_allclose(b, a[perm], rtol=1e-13, atol=1e-16)


# --- keep counts: ceil((1-P)|S|) of Eq. (inner) -------------------------------------------

def test_keep_count_rule_closed_forms():
    kc = oracle.keep_count
    assert math.ceil(0.55 * 100) == 56            # the floating-point trap
    assert kc(0.55, 100) == 55 and kc(0.55, 3000) == 1650
    assert kc(0.7, 3000) == 2100
    assert kc(0.5, 250) == 125 and kc(0.3, 1000) == 300
    assert kc(0.3, 1001) == 301                   # 300.3 -> 301
    assert kc(0.0, 10) == 0 and kc(1.0, 10) == 10 and kc(0.5, 0) == 0
    assert kc(0.001, 1) == 1                      # any positive fraction keeps one
    with pytest.raises(ValueError):
        kc(1.5, 10)


def test_keep_counts_of_the_workloads():
    """Token counts after each step, derived by hand from the workload
    definitions: kept = system + query + ceil(r_a N_a) + ceil(r_v N_v)."""
    from synth import workload
    from synth.inputs import base_counts
    expect = {
        "tiny": [16 + 32 + 125 + 300],                      # 250*.5, 1000*.3
        "3b_60s": [16 + 64 + 750 + 1800],                   # 1500*.5, 7200*.25
        "7b_2min": [16 + 128 + 2100 + 9600, 16 + 128 + 1500 + 6000, 16 + 128 + 900 + 3600],
        "7b_10min": [16 + 256 + 10500 + 48000, 16 + 256 + 7500 + 30000, 16 + 256 + 4500 + 18000],
    }
    assert expect["tiny"] == [473] and expect["3b_60s"] == [2630]
    assert expect["7b_2min"] == [11844, 7644, 4644] and expect["7b_10min"] == [58772, 37772, 22772]
    for name, totals in expect.items():
        wl = workload(name)
        for step, total in enumerate(totals):
            counts = oracle.step_keep_counts(wl.ratios[step], base_counts(wl))
            got = sum(s.n_sys + s.n_q + a + v for s, (a, v) in zip(wl.seqs, counts))
            assert got == total, (name, step)


# --- selection -----------------------------------------------------------------------------

@pytest.mark.parametrize("joint", [False, True])
def test_selection_matches_rank_counting_brute_force(joint):
    rng = np.random.default_rng(7)
    mod = np.concatenate([rng.choice([0, 1, 2], 40, p=[0.2, 0.3, 0.5]),
                          rng.choice([0, 1, 2], 25, p=[0.1, 0.5, 0.4])]).astype(np.uint8)
    cu = np.array([0, 40, 65], np.int32)
    scores = rng.integers(0, 6, mod.size).astype(np.float64) / 7.0   # many ties
    scores[mod == 0] = 0
    counts = []
    for s in range(2):
        m = mod[cu[s]:cu[s + 1]]
        na, nv = int((m == 1).sum()), int((m == 2).sum())
        counts.append(((na + nv) // 2, 0) if joint else (na // 2, (nv * 2) // 3))
    got = oracle.select_keep(scores, mod, cu, counts, joint=joint)
    ref = brute_select(scores, mod, cu, counts, joint=joint)
    np.testing.assert_array_equal(got, ref)


def test_selection_invariants_and_ties_to_lower_index():
    mod = np.array([0, 1, 2, 1, 2, 2, 1, 0, 2, 0], np.uint8)
    cu, _ = one_seq(mod)
    scores = np.where(mod == 0, 0.0, 0.25)           # all equal within S
    keep = oracle.select_keep(scores, mod, cu, [(2, 2)])
    np.testing.assert_array_equal(keep, [0, 1, 2, 3, 4, 7, 9])
    keep = oracle.select_keep(scores, mod, cu, [(0, 4)])
    np.testing.assert_array_equal(keep, [0, 2, 4, 5, 7, 8, 9])
    keep = oracle.select_keep(scores, mod, cu, [(3, 0)])
    np.testing.assert_array_equal(keep, [0, 1, 3, 6, 7, 9])
    with pytest.raises(ValueError):
        oracle.select_keep(scores, mod, cu, [(4, 0)])


def test_planted_tokens_are_kept_on_the_tiny_workload():
    from synth import workload
    from synth.inputs import query_rows, key_slab, planted_tokens, base_counts
    wl = workload("tiny")
    q = query_rows(wl, 0)
    k = key_slab(wl, 0, q)
    mod = wl.modality()
    out = oracle.prune_step(q, k, wl.cu_seqlens(), wl.cu_qlens(), mod, wl.num_q_heads,
                            wl.num_kv_heads, oracle.step_keep_counts(wl.ratios[0], base_counts(wl)))
    tok, _ = planted_tokens(wl)
    assert tok.size == 28
    assert np.isin(tok, out["keep_idx"]).all()
    keep = out["keep_idx"]
    assert keep.size == 473 and np.all(np.diff(keep) > 0)
    assert np.isin(np.nonzero(mod == 0)[0], keep).all()
    # margin: every plant beats the k-th kept score of its modality
    sc = out["scores"]
    for m in (1, 2):
        kept_m = keep[mod[keep] == m]
        kth = sc[kept_m].min()
        pm = tok[mod[tok] == m]
        assert sc[pm].min() > kth


# --- compaction ----------------------------------------------------------------------------

def test_compaction_row_by_row_and_progressive_composition():
    rng = np.random.default_rng(8)
    T = 37
    plane = rng.integers(0, 2 ** 16, (T, 24), dtype=np.uint16)
    mod = rng.choice([0, 1, 2], T).astype(np.uint8)
    cu = np.array([0, 20, T], np.int32)
    scores = rng.random(T)
    k1 = oracle.select_keep(scores, mod, cu, [(3, 4), (2, 3)])
    out1 = oracle.compact_rows(plane, k1)
    for j, i in enumerate(k1):                      # byte-for-byte, row by row
        assert out1[j].tobytes() == plane[i].tobytes()
    cu1 = oracle.new_cu_seqlens(k1, cu)
    assert cu1.tolist() == [0, int((k1 < 20).sum()), k1.size]
    mod1 = oracle.compact_rows(mod, k1)
    k2 = oracle.select_keep(scores[k1], mod1, cu1, [(1, 2), (1, 1)])
    out2 = oracle.compact_rows(out1, k2)
    np.testing.assert_array_equal(out2, oracle.compact_rows(plane, k1[k2]))


# ---------------------------------------------------------------- causal-row softmax domain

def brute_scores_causal(q_bits, k_bits, cu, cuq, mod, Hq, Hkv, q_start=None):
    """Arbitrary-precision reference of the causal-row domain: query row r of a
    sequence of length L is token p = q_start + r (q_start = L - n_q when not
    given); its softmax runs over tokens 0..p of the sequence (every modality),
    explicit loops at 40 digits."""
    mpmath.mp.dps = 40
    q = oracle.bf16_to_f64(q_bits)
    k = oracle.bf16_to_f64(k_bits)
    T = k.shape[0]
    out = [mpmath.mpf(0)] * T
    g = Hq // Hkv
    for s in range(len(cu) - 1):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        nq = int(cuq[s + 1] - cuq[s])
        if nq == 0 or not any(mod[i] in (1, 2) for i in range(t0, t1)):
            continue
        for h in range(Hq):
            for r in range(nq):
                pos = (t1 - t0 - nq if q_start is None else int(q_start[s])) + r
                vis = range(t0, t0 + pos + 1)
                logits = {i: mpmath.fsum(mpmath.mpf(float(a)) * mpmath.mpf(float(b))
                                         for a, b in zip(q[cuq[s] + r, h], k[i, h // g])) / mpmath.sqrt(D)
                          for i in vis}
                z = mpmath.fsum(mpmath.exp(x) for x in logits.values())
                for i in vis:
                    if mod[i] in (1, 2):
                        out[i] += mpmath.exp(logits[i]) / z
        for i in range(t0, t1):
            out[i] /= Hq * nq
    return np.array([float(v) for v in out])


@pytest.mark.parametrize("Hq,Hkv,nq", [(4, 2, 3), (2, 2, 1), (6, 1, 4)])
def test_causal_scores_match_arbitrary_precision_brute_force(Hq, Hkv, nq):
    rng = np.random.default_rng(100 + Hq * 10 + Hkv)
    # the second sequence has tokens of S among its last rows (inside the query span)
    mod = np.array([0, 0, 1, 2, 2, 1, 2, 2, 2, 1, 0, 2, 1, 1, 0, 0], np.uint8)
    mod2 = np.array([0, 2, 2, 1, 2, 1, 0, 2, 0, 1], np.uint8)
    modality = np.concatenate([mod, mod2])
    cu = np.array([0, mod.size, modality.size], np.int32)
    cuq = np.array([0, nq, 2 * nq], np.int32)
    k = rand_bf16(rng, (modality.size, Hkv, D))
    q = rand_bf16(rng, (2 * nq, Hq, D), 0.3)
    got = oracle.relevance_scores(q, k, cu, cuq, modality, Hq, Hkv, softmax_domain=oracle.SOFTMAX_CAUSAL_ROW)
    ref = brute_scores_causal(q, k, cu, cuq, modality, Hq, Hkv)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-15)
    assert np.all(got[modality == 0] == 0)


@pytest.mark.parametrize("Hq,Hkv,nq", [(4, 2, 3), (6, 1, 4)])
def test_causal_scores_with_the_query_span_inside_the_sequence(Hq, Hkv, nq):
    # the query rows start at a given position (tokens after the span are seen by no row)
    rng = np.random.default_rng(300 + Hq + nq)
    mod = np.array([0, 0, 1, 2, 2, 1, 2, 2, 2, 1, 0, 2, 1, 1, 0, 0], np.uint8)
    mod2 = np.array([0, 2, 2, 1, 2, 1, 0, 2, 0, 1], np.uint8)
    modality = np.concatenate([mod, mod2])
    cu = np.array([0, mod.size, modality.size], np.int32)
    cuq = np.array([0, nq, 2 * nq], np.int32)
    q_start = np.array([5, 2], np.int32)
    k = rand_bf16(rng, (modality.size, Hkv, D))
    q = rand_bf16(rng, (2 * nq, Hq, D), 0.3)
    got = oracle.relevance_scores(q, k, cu, cuq, modality, Hq, Hkv, softmax_domain=oracle.SOFTMAX_CAUSAL_ROW,
                                  q_start=q_start)
    ref = brute_scores_causal(q, k, cu, cuq, modality, Hq, Hkv, q_start=q_start)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-15)
    # tokens after the last row's position get nothing
    assert np.all(got[q_start[0] + nq:mod.size] == 0)
    assert np.all(got[mod.size + q_start[1] + nq:] == 0)
    # the default is the span at the end of each sequence
    end = oracle.relevance_scores(q, k, cu, cuq, modality, Hq, Hkv, softmax_domain=oracle.SOFTMAX_CAUSAL_ROW,
                                  q_start=np.diff(cu) - nq)
    np.testing.assert_array_equal(end, oracle.relevance_scores(q, k, cu, cuq, modality, Hq, Hkv,
                                                               softmax_domain=oracle.SOFTMAX_CAUSAL_ROW))


def test_causal_identical_keys_closed_form():
    # Identical keys: every visible token has the same logit, so row r spreads its
    # mass uniformly over the p_r + 1 tokens it sees (every modality, itself
    # included), p_r = L - n_q + r; a token of S at position i collects
    # (1/n_q) sum over rows with p_r >= i of 1/(p_r + 1).
    rng = np.random.default_rng(5)
    L, nq, Hq, Hkv = 23, 5, 4, 2
    mod = np.zeros(L, np.uint8)
    mod[[1, 2, 5, 8, 9, 13]] = 1
    mod[[3, 4, 10, 11, 16]] = 2
    mod[[19, 21]] = 2                       # inside the query span (positions 18..22)
    k = np.repeat(rand_bf16(rng, (1, Hkv, D)), L, axis=0)
    q = rand_bf16(rng, (nq, Hq, D))
    cu, _ = one_seq(mod)
    got = oracle.relevance_scores(q, k, cu, np.array([0, nq]), mod, Hq, Hkv,
                                  softmax_domain=oracle.SOFTMAX_CAUSAL_ROW)
    for i in range(L):
        want = 0.0
        if mod[i]:
            want = sum(1.0 / (L - nq + r + 1) for r in range(nq) if L - nq + r >= i) / nq
        assert got[i] == pytest.approx(want, rel=1e-13, abs=0.0), i
    # the mass on the non-S tokens (system, text, query rows) is what S loses
    assert got.sum() < 1.0


def test_causal_domain_reduces_to_the_S_domain_when_other_keys_are_negligible():
    # One head, one query row (the last token).  Keys outside S point against the
    # query (logit about -40, against logits of order 1 on S), so their share is
    # below 1e-16: the causal-row scores equal the S-domain scores, which equal
    # scipy's softmax over S.
    rng = np.random.default_rng(6)
    L = 40
    mod = np.full(L, 1, np.uint8)
    mod[[0, 1, 2, 20, 39]] = 0
    q = np.zeros((1, 1, D), np.float32)
    q[0, 0, :] = rng.standard_normal(D).astype(np.float32)
    k = rng.standard_normal((L, 1, D)).astype(np.float32) * 0.5
    u = q[0, 0] / np.linalg.norm(q[0, 0])
    k[mod == 0, 0, :] = -40.0 * u
    qb, kb = bf16(q), bf16(k)
    cu, _ = one_seq(mod)
    causal = oracle.relevance_scores(qb, kb, cu, np.array([0, 1]), mod, 1, 1,
                                     softmax_domain=oracle.SOFTMAX_CAUSAL_ROW)
    mm = oracle.relevance_scores(qb, kb, cu, np.array([0, 1]), mod, 1, 1)
    np.testing.assert_allclose(causal, mm, rtol=1e-12, atol=0)
    S = np.nonzero(mod)[0]
    ref = scipy.special.softmax(oracle.bf16_to_f64(kb)[S, 0, :] @ oracle.bf16_to_f64(qb)[0, 0, :] / np.sqrt(D))
    np.testing.assert_allclose(causal[S], ref, rtol=1e-12)
