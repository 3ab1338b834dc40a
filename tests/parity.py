"""Comparison rules between the CUDA path and the oracle.

Scores: |gpu - oracle| <= 1e-5 + 2e-3 |oracle| (fp32 accumulation of bf16
products against fp64).  Kept indices: identical, except tokens whose oracle
score lies within that tolerance of the k-th kept score of their segment
(the two sides may order such near-ties differently).  Compacted rows:
bit-exact given the GPU's own indices.
"""

import numpy as np

import oracle


def check_scores(gpu, ref, strict_rel=None):
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


def check_keep(gpu_keep, ref_keep, ref_scores, modality, cu, joint=False):
    """Returns the number of tie-exempt tokens; raises on any other difference."""
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
        tol = 1e-5 + 2e-3 * abs(kth)
        far = diff[np.abs(ref_scores[diff] - kth) > tol]
        assert far.size == 0, f"tokens {far[:5]} differ and are not near the k-th score {kth}"
        exempt += diff.size
    return exempt
