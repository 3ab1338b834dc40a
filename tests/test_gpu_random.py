"""Randomised end-to-end prune steps (apack_prune_step: score, select, compact) against the
oracle: ragged batches with empty sequences, sequences without S or without query rows, one to
three hundred query rows (so both scoring paths run), four head layouts, both softmax domains,
per-modality and joint selection, keep ratios including 0 and 1.

Per step: scores under the strict and the graded rule, kept indices equal to the oracle's up to
ties inside the measured error band, offsets and compacted K/V/hidden rows bit-exact for the
GPU's own indices (Sec. 3.2, Eq. inner_score and Eq. inner; Algorithm 1, "slice their KV-cache
entries").
"""

import numpy as np
import pytest
import torch

import oracle
from parity import check_scores, check_keep
from synth.gen import f32_to_bf16_bits

pytestmark = pytest.mark.gpu

D = 128
HEADS = [(28, 4), (16, 2), (8, 8), (12, 2)]


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


def draw_case(rng):
    hq, hkv = HEADS[int(rng.integers(len(HEADS)))]
    B = int(rng.integers(1, 6))
    lens, nqs = [], []
    for _ in range(B):
        L = 0 if rng.random() < 0.1 else int(rng.integers(1, 3000))
        nq = int(rng.choice([0, 1, 2, int(rng.integers(1, 300)), int(rng.integers(1, 300))]))
        lens.append(L)
        nqs.append(min(nq, L))                 # the query span lies inside its sequence
    mods = []
    for L in lens:
        if rng.random() < 0.1:                 # a sequence without S
            mods.append(np.zeros(L, np.uint8))
            continue
        m = rng.choice([1, 2], L, p=[0.25, 0.75]).astype(np.uint8)
        m[rng.random(L) < rng.uniform(0.0, 0.2)] = 0
        mods.append(m)
    mod = np.concatenate(mods) if mods else np.zeros(0, np.uint8)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    cuq = np.concatenate([[0], np.cumsum(nqs)]).astype(np.int32)
    domain = int(rng.integers(2))
    joint = bool(rng.integers(2))
    ratios = rng.uniform(0.0, 1.0, (B, 2))
    ratios[rng.random((B, 2)) < 0.15] = 0.0
    ratios[rng.random((B, 2)) < 0.15] = 1.0
    return hq, hkv, lens, nqs, mod, cu, cuq, domain, joint, np.round(ratios, 3)


@pytest.mark.parametrize("seed", range(40))
def test_random_prune_step_matches_oracle(ap, seed):
    rng = np.random.default_rng(1000 + seed)
    hq, hkv, lens, nqs, mod, cu, cuq, domain, joint, ratios = draw_case(rng)
    T, NQ = int(cu[-1]), int(cuq[-1])
    B = len(lens)
    na = [int((mod[cu[s]:cu[s + 1]] == 1).sum()) for s in range(B)]
    nv = [int((mod[cu[s]:cu[s + 1]] == 2).sum()) for s in range(B)]
    k_bits = f32_to_bf16_bits((rng.standard_normal((T, hkv, D)) * 1.4).astype(np.float32))
    q_bits = f32_to_bf16_bits(rng.standard_normal((max(NQ, 1), hq, D)).astype(np.float32))[:NQ]
    L_layers, layer, H = 3, 1, 256
    nl, row = L_layers - layer, hkv * D * 2
    kc = torch.from_numpy(rng.integers(-30000, 30000, (nl, T, row // 2), dtype=np.int16)).cuda()
    kc[0] = dev(k_bits).view(T, row // 2)
    vc = torch.from_numpy(rng.integers(-30000, 30000, (nl, T, row // 2), dtype=np.int16)).cuda()
    hid = torch.from_numpy(rng.integers(-30000, 30000, (T, H), dtype=np.int16)).cuda()

    mode = ap.APACK_SELECT_JOINT if joint else ap.APACK_SELECT_PER_MODALITY
    if joint:
        counts = [(oracle.keep_count(float(ratios[s, 0]), na[s] + nv[s]), 0) for s in range(B)]
    else:
        counts = [(oracle.keep_count(float(ratios[s, 0]), na[s]), oracle.keep_count(float(ratios[s, 1]), nv[s]))
                  for s in range(B)]
    n_out = T - sum(na) - sum(nv) + sum(a + b for a, b in counts)

    seqs = ap.Seqs(cu, cuq, na, nv, dev(mod), hq, hkv, softmax_domain=domain)
    n_ws = ap.apack_workspace_size(seqs)
    ws_t = torch.zeros(n_ws + 256, dtype=torch.uint8, device="cuda")
    off = (-ws_t.data_ptr()) % 256
    ws = ws_t[off:off + n_ws]
    keep = torch.empty(max(n_out, 1), dtype=torch.int32, device="cuda")
    mod_out = torch.empty(max(n_out, 1), dtype=torch.uint8, device="cuda")
    scores = torch.empty(max(T, 1), dtype=torch.float32, device="cuda")
    ko = torch.empty((nl, max(n_out, 1), row // 2), dtype=torch.int16, device="cuda")
    vo = torch.empty_like(ko)
    ho = torch.empty((max(n_out, 1), H), dtype=torch.int16, device="cuda")
    q_d = dev(q_bits) if NQ else torch.zeros(16, dtype=torch.int16, device="cuda")
    new_cu = ap.apack_prune_step(seqs, layer, L_layers, q_d, kc, vc, T * row, hid, H, keep_ratio=ratios,
                                 select_mode=mode, k_out=ko, v_out=vo, kv_out_layer_stride=max(n_out, 1) * row,
                                 hidden_out=ho, modality_out=mod_out, keep_idx=keep, scores=scores, ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK

    ref_scores = oracle.relevance_scores(q_bits, k_bits, cu, cuq, mod, hq, hkv, softmax_domain=domain)
    got_scores = scores[:T].cpu().numpy()
    max_rel = check_scores(got_scores, ref_scores)
    ref_keep = oracle.select_keep(ref_scores, mod, cu, counts, joint=joint)
    got_keep = keep[:n_out].cpu().numpy().astype(np.int64)
    check_keep(got_keep, ref_keep, ref_scores, mod, cu, joint=joint, rel_band=2.01 * max_rel + 1e-12)
    # selection is exact on the GPU's own scores; offsets and rows follow the GPU's indices
    np.testing.assert_array_equal(got_keep, oracle.select_keep(got_scores, mod, cu, counts, joint=joint))
    np.testing.assert_array_equal(new_cu, oracle.new_cu_seqlens(got_keep, cu))
    np.testing.assert_array_equal(mod_out[:n_out].cpu().numpy(), oracle.compact_rows(mod, got_keep))
    kn, vn, hn = kc.cpu().numpy(), vc.cpu().numpy(), hid.cpu().numpy()
    for li in range(nl):
        np.testing.assert_array_equal(ko[li, :n_out].cpu().numpy(), oracle.compact_rows(kn[li], got_keep))
        np.testing.assert_array_equal(vo[li, :n_out].cpu().numpy(), oracle.compact_rows(vn[li], got_keep))
    np.testing.assert_array_equal(ho[:n_out].cpu().numpy(), oracle.compact_rows(hn, got_keep))


def draw_keep(rng, T, n_keep):
    """Strictly increasing kept rows of one of four shapes (uniform, kept prefix, kept tail, runs)."""
    kind = int(rng.integers(4))
    if kind == 0 or n_keep in (0, T):
        return np.sort(rng.choice(T, n_keep, replace=False))
    if kind == 1:      # a prefix that stays in place, then a uniform choice
        head = int(rng.integers(0, n_keep + 1))
        rest = np.sort(rng.choice(np.arange(head, T), n_keep - head, replace=False))
        return np.concatenate([np.arange(head), rest])
    if kind == 2:      # a uniform choice, then the whole tail
        tail = int(rng.integers(0, n_keep + 1))
        head = np.sort(rng.choice(T - tail, n_keep - tail, replace=False))
        return np.concatenate([head, np.arange(T - tail, T)])
    starts = np.sort(rng.choice(T, min(T, max(1, n_keep // 37)), replace=False))   # runs of kept rows
    keep = np.unique(np.concatenate([np.arange(s, min(T, s + 64)) for s in starts]))
    if keep.size >= n_keep:
        return np.sort(rng.choice(keep, n_keep, replace=False))
    extra = rng.choice(np.setdiff1d(np.arange(T), keep), n_keep - keep.size, replace=False)
    return np.sort(np.concatenate([keep, extra]))


@pytest.mark.parametrize("seed", range(24))
def test_random_in_place_compaction_matches_oracle(ap, seed):
    """apack_compact with src == dst on random keep lists of every density (the wave schedule for
    low keep ratios, the per-item one near 1), one to three groups of various row sizes."""
    rng = np.random.default_rng(5000 + seed)
    T = int(rng.integers(1, 40000))
    n_keep = int(rng.integers(0, T + 1)) if rng.random() < 0.8 else int(T * rng.uniform(0.8, 1.0))
    keep = draw_keep(rng, T, n_keep).astype(np.int32)
    assert keep.size == n_keep
    shapes = [(int(rng.integers(1, 4)), int(rng.choice([16, 256, 1024, 2048, 7168])))
              for _ in range(int(rng.integers(1, 4)))]
    while T * sum(pl * rb for pl, rb in shapes) > 400_000_000:      # a few hundred MB per case
        shapes = shapes[:-1] if len(shapes) > 1 else [(1, shapes[0][1])]
    srcs = [rng.integers(0, 256, (pl, T, rb), dtype=np.uint8) for pl, rb in shapes]
    bufs = [dev(s) for s in srcs]
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    groups = [ap.make_plane(b, b, rb, pl, src_plane_stride=T * rb, dst_plane_stride=T * rb)
              for b, (pl, rb) in zip(bufs, shapes)]
    if n_keep:
        ap.apack_compact(dev(keep), n_keep, groups, ws=ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    for b, s in zip(bufs, srcs):
        got = b.cpu().numpy()
        for pl in range(s.shape[0]):
            np.testing.assert_array_equal(got[pl, :n_keep], oracle.compact_rows(s[pl], keep))
            np.testing.assert_array_equal(got[pl, n_keep:], s[pl, n_keep:])
