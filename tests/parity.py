"""Comparison rules between the CUDA path and the oracle.

Scores: |gpu - oracle| <= 1e-5 + 2e-3 |oracle| (the graded rule: fp32
accumulation of bf16 products against fp64), and by default also the strict
relative-only rule |gpu - oracle| <= 2e-3 |oracle| on every token of S.  At
10^5 tokens a typical score is about 1/|S| < 1e-5, below the graded rule's
absolute term, so only the strict rule says anything there.

Kept indices: identical, except tokens whose oracle score lies near the k-th
kept score of their segment (the two sides may order such near-ties
differently).  With `rel_band` set, "near" is |I - I_k| <= rel_band |I_k|: a
GPU whose scores carry relative error e can swap two tokens only if both lie
within about 2e |I_k| of the k-th score, so rel_band = 2e (e measured) leaves
no room for a swap that the score error does not explain.  Compacted rows:
bit-exact given the GPU's own indices.
"""

import numpy as np

import oracle


STRICT_REL = 2e-3


def check_scores(gpu, ref, strict_rel=STRICT_REL):
    """Asserts both rules; returns the largest relative error over the tokens of S."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    tol = oracle.score_tolerance(ref)
    bad = np.nonzero(np.abs(gpu - ref) > tol)[0]
    assert bad.size == 0, f"{bad.size} scores out of tolerance, first {bad[:5]}: {gpu[bad[:5]]} vs {ref[bad[:5]]}"
    if strict_rel is not None:
        rel = np.abs(gpu - ref) / np.maximum(np.abs(ref), 1e-300)
        mm = ref > 0
        assert rel[mm].max(initial=0) <= strict_rel, f"max rel err {rel[mm].max()}"
    rel = np.abs(gpu - ref) / np.maximum(np.abs(ref), 1e-30)
    return float(rel[ref > 0].max(initial=0.0))


def segments(modality, cu, joint=False):
    """Yields (mask of segment tokens) per (sequence, modality)."""
    T = modality.size
    for s in range(len(cu) - 1):
        inseq = np.zeros(T, bool)
        inseq[cu[s]:cu[s + 1]] = True
        if joint:
            yield inseq & ((modality == 1) | (modality == 2))
        else:
            yield inseq & (modality == 1)
            yield inseq & (modality == 2)


def check_keep(gpu_keep, ref_keep, ref_scores, modality, cu, joint=False, rel_band=None):
    """Returns the number of tokens kept by one side only (all of them near-ties);
    raises on any other difference.  rel_band None: the graded rule's band."""
    gpu_keep = np.asarray(gpu_keep, np.int64)
    ref_keep = np.asarray(ref_keep, np.int64)
    assert gpu_keep.size == ref_keep.size
    assert np.all(np.diff(gpu_keep) > 0), "keep_idx not strictly increasing"
    other = np.nonzero((modality != 1) & (modality != 2))[0]
    assert np.isin(other, gpu_keep).all(), "a token outside S was dropped"
    if np.array_equal(gpu_keep, ref_keep):
        return 0
    kg = np.zeros(modality.size, bool); kg[gpu_keep] = True
    kr = np.zeros(modality.size, bool); kr[ref_keep] = True
    exempt = 0
    for seg in segments(modality, cu, joint):
        g, r = kg & seg, kr & seg
        assert g.sum() == r.sum(), "kept count differs in a segment"
        diff = np.nonzero(g ^ r)[0]
        if diff.size == 0:
            continue
        kth = ref_scores[np.nonzero(r)[0]].min()
        tol = 1e-5 + 2e-3 * abs(kth) if rel_band is None else rel_band * abs(kth)
        far = diff[np.abs(ref_scores[diff] - kth) > tol]
        assert far.size == 0, f"tokens {far[:5]} differ and are not near the k-th score {kth}"
        exempt += diff.size
    return exempt


def tie_bands(ref_scores, ref_keep, modality, cu, joint=False):
    """Tokens of S that each rule would let the two sides order differently: those whose
    oracle score lies within the rule's tolerance of their segment's k-th kept score.
    Returns (graded, strict) counts summed over segments."""
    kr = np.zeros(modality.size, bool)
    kr[np.asarray(ref_keep, np.int64)] = True
    graded = strict = 0
    for seg in segments(modality, cu, joint):
        kept = np.nonzero(kr & seg)[0]
        if kept.size == 0 or kept.size == seg.sum():
            continue
        kth = ref_scores[kept].min()
        d = np.abs(ref_scores[seg] - kth)
        graded += int((d <= 1e-5 + 2e-3 * abs(kth)).sum())
        strict += int((d <= STRICT_REL * abs(kth)).sum())
    return graded, strict
