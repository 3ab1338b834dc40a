"""apack_score_static: scoring for callers that cannot allocate device memory.

Some callers cannot call cudaMalloc: a plugin inside an inference engine that
owns every device allocation, or a server that fixes its device memory at
start-up so that no request can fail on an allocation.  For them the library
keeps one fixed 8 MiB scratch array per device instead of a caller workspace.

These checks call it through the C ABI and compare its scores with those of
apack_score (which gets an ordinary workspace), on consecutive calls: the
array keeps the previous call's contents, so each call must start clean.
"""

import numpy as np
import pytest
import torch

from parity import check_scores

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def _inputs(ap, name, duration_s=None):
    from synth import workload
    from synth.configs import scaled_copy
    from synth.inputs import query_rows, key_slab
    wl = workload(name)
    if duration_s is not None:
        wl = scaled_copy(wl, duration_s)
    layer = wl.prune_layers[0]
    q = query_rows(wl, layer)
    k = key_slab(wl, layer, q)
    mod = torch.from_numpy(wl.modality()).cuda()
    seqs = ap.Seqs(wl.cu_seqlens(), wl.cu_qlens(), [s.n_audio for s in wl.seqs], [s.n_visual for s in wl.seqs],
                   mod, wl.num_q_heads, wl.num_kv_heads)
    q_d = torch.from_numpy(q.view(np.int16)).cuda()
    k_d = torch.from_numpy(k.view(np.int16)).cuda()
    return seqs, q_d, k_d, wl.num_kv_heads * wl.head_dim * 2, wl.total_tokens, mod


def _with_workspace(ap, seqs, q, k, stride, T):
    n = ap.apack_workspace_size(seqs)
    ws = torch.zeros(n + 256, dtype=torch.uint8, device="cuda")
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + n]
    out = torch.empty(T, dtype=torch.float32, device="cuda")
    ap.apack_score(seqs, q, k, stride, out, ws)
    torch.cuda.synchronize()
    assert ap.apack_device_error(ws) == ap.APACK_OK
    return out.cpu().numpy()


def _static(ap, seqs, q, k, stride, T):
    out = torch.full((T,), float("nan"), dtype=torch.float32, device="cuda")
    err = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    ap.apack_score_static(seqs, q, k, stride, out, device_error_out=err)
    torch.cuda.synchronize()
    assert int(err.item()) == ap.APACK_OK
    return out.cpu().numpy()


def test_static_scratch_matches_workspace_scores_on_consecutive_calls(ap):
    a = _inputs(ap, "7b_2min")
    b = _inputs(ap, "tiny")
    # the paper's own setting (last query token only) on a 200-s sequence: the few-row
    # scoring path, which lays the scratch array out differently (logits, per-CTA partials)
    p = _inputs(ap, "7b_10min_paper", duration_s=200)
    ref_a = _with_workspace(ap, *a[:5])
    ref_b = _with_workspace(ap, *b[:5])
    ref_p = _with_workspace(ap, *p[:5])
    # two calls in a row on the same batch, then other batches, the two scoring paths
    # interleaved, each reading an array the other layout wrote last
    for args, ref in ((a, ref_a), (a, ref_a), (p, ref_p), (b, ref_b), (p, ref_p), (p, ref_p), (a, ref_a)):
        got = _static(ap, *args[:5])
        check_scores(got, ref)
        assert np.array_equal(got, ref)   # same kernels, same order: bit for bit


def test_static_scratch_rejects_batches_over_its_limit(ap):
    big = _inputs(ap, "7b_ragged16")      # needs about 43 MiB of scratch
    seqs, q, k, stride, T, _ = big
    out = torch.zeros(T, dtype=torch.float32, device="cuda")
    with pytest.raises(ap.ApackError) as e:
        ap.apack_score_static(seqs, q, k, stride, out)
    assert e.value.status == ap.APACK_EWORKSPACE
    assert not out.any()


def test_static_scratch_refuses_host_keys_before_any_device_work(ap):
    # the keys are read by TMA, so pinned host memory is refused as apack_score
    # refuses it, and nothing is written
    seqs, q, k, stride, T, _ = _inputs(ap, "tiny")
    out = torch.zeros(T, dtype=torch.float32, device="cuda")
    k_host = k.cpu().pin_memory()
    with pytest.raises(ap.ApackError) as e:
        ap.apack_score_static(seqs, q, k_host, stride, out)
    assert e.value.status == ap.APACK_EINVAL
    torch.cuda.synchronize()
    assert not out.any()
