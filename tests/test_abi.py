"""The C ABI on the host: the library loads, exports every entry point that
include/apack.h declares, validates arguments before touching the device and
computes keep counts by the rule of Eq. inner (checked against the oracle).
No CUDA compute is launched here."""

import ctypes
import os
import re

import numpy as np
import pytest

import oracle

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def ap():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2608_08794_gb300 as ap
    return ap


def declared_functions():
    text = open(os.path.join(ROOT, "include", "apack.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(apack_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(ap):
    names = declared_functions()
    assert set(names) >= {"apack_score", "apack_select", "apack_compact", "apack_prune_step",
                          "apack_workspace_size", "apack_keep_counts", "apack_device_error"}
    lib = ctypes.CDLL(ap.library_path())
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(ap.EXPORTED)


def make_seqs(ap, lens=(40, 25), nq=(3, 2), na=(10, 5), nv=(20, 12), hq=28, hkv=4, head_dim=128):
    cu = np.concatenate([[0], np.cumsum(lens)])
    cuq = np.concatenate([[0], np.cumsum(nq)])
    return ap.Seqs(cu, cuq, na, nv, None, hq, hkv, head_dim)


def test_workspace_size_and_validation(ap):
    s = make_seqs(ap)
    s.struct.modality = 0x1000          # a non-null placeholder; nothing is dereferenced on the host
    n = ap.apack_workspace_size(s)
    assert n > 0 and n % 256 == 0
    bad = make_seqs(ap, hq=28, hkv=3)
    bad.struct.modality = 0x1000
    with pytest.raises(ap.ApackError) as e:
        ap.apack_workspace_size(bad)
    assert e.value.status == ap.APACK_EINVAL
    bad = make_seqs(ap, head_dim=64)
    bad.struct.modality = 0x1000
    with pytest.raises(ap.ApackError) as e:
        ap.apack_workspace_size(bad)
    assert e.value.status == ap.APACK_EUNSUPPORTED
    bad = make_seqs(ap, na=(30, 5))     # more MM tokens than the sequence holds
    bad.struct.modality = 0x1000
    with pytest.raises(ap.ApackError):
        ap.apack_workspace_size(bad)
    bad = make_seqs(ap)                  # T > 0 but no modality pointer
    with pytest.raises(ap.ApackError):
        ap.apack_workspace_size(bad)


def test_keep_counts_match_oracle_rule(ap):
    rng = np.random.default_rng(0)
    B = 64
    lens = rng.integers(0, 5000, B)
    na = (lens * rng.random(B) * 0.3).astype(int)
    nv = ((lens - na) * rng.random(B) * 0.9).astype(int)
    s = make_seqs(ap, lens=lens, nq=np.ones(B, int), na=na, nv=nv)
    s.struct.modality = 0x1000
    ratios = np.round(rng.random((B, 2)), 3).astype(np.float32)
    ratios[:4] = [[0.55, 0.55], [0.0, 1.0], [1.0, 0.0], [0.7, 0.15]]
    k, cu = ap.apack_keep_counts(s, ratios)
    for b in range(B):
        assert k[b, 0] == oracle.keep_count(float(ratios[b, 0]), na[b])
        assert k[b, 1] == oracle.keep_count(float(ratios[b, 1]), nv[b])
    assert cu[0] == 0 and np.all(np.diff(cu) == lens - na - nv + k[:, 0] + k[:, 1])
    kj, _ = ap.apack_keep_counts(s, ratios, ap.APACK_SELECT_JOINT)
    for b in range(B):
        assert kj[b, 0] == oracle.keep_count(float(ratios[b, 0]), na[b] + nv[b]) and kj[b, 1] == 0
    with pytest.raises(ap.ApackError):
        ap.apack_keep_counts(s, np.full((B, 2), 1.5, np.float32))


def test_calls_reject_bad_arguments_before_the_device(ap):
    import torch  # noqa: F401  (CPU tensors only: pointers are never dereferenced)
    s = make_seqs(ap)
    s.struct.modality = 0x1000
    ws_small = torch.zeros(256, dtype=torch.uint8)
    with pytest.raises(ap.ApackError) as e:
        ap.apack_score(s, ws_small, ws_small, 1024, ws_small, ws_small, stream=0)
    assert e.value.status == ap.APACK_EWORKSPACE
    # the fixed-scratch scorer checks its pointers before it touches a device
    with pytest.raises(ap.ApackError) as e:
        ap.apack_score_static(s, None, ws_small, 1024, ws_small, stream=0)
    assert e.value.status == ap.APACK_EINVAL
    with pytest.raises(ap.ApackError) as e:
        ap.apack_select(s, ws_small, np.array([[11, 0], [0, 0]]), ws_small, ws_small, stream=0)
    assert e.value.status in (ap.APACK_EINVAL, ap.APACK_EWORKSPACE)
    # count larger than the segment
    ws = torch.zeros(ap.apack_workspace_size(s) + 256, dtype=torch.uint8)
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + ap.apack_workspace_size(s)]
    with pytest.raises(ap.ApackError) as e:
        ap.apack_select(s, ws_small, np.array([[11, 0], [0, 0]]), ws_small, ws, stream=0)
    assert e.value.status == ap.APACK_EINVAL
    # in-place compaction: needs the workspace's progress words, vector rows and one layout
    t = torch.zeros(4096, dtype=torch.uint8)
    p = ap.make_plane(t, t, 256)
    with pytest.raises(ap.ApackError) as e:
        ap.apack_compact(t, 4, [p], stream=0)
    assert e.value.status == ap.APACK_EINVAL
    with pytest.raises(ap.ApackError) as e:
        ap.apack_compact(t, 4, [ap.make_plane(t, t, 40)], ws=ws, stream=0)
    assert e.value.status == ap.APACK_EUNSUPPORTED
    with pytest.raises(ap.ApackError) as e:
        ap.apack_compact(t, 4, [ap.make_plane(t, t, 256, 2, 1024, 512)], ws=ws, stream=0)
    assert e.value.status == ap.APACK_EINVAL
    assert ap.status_string(ap.APACK_ETIMEOUT) == "device wait timed out"


def test_step_and_schedule_check_their_compaction_before_any_launch(ap):
    # A bad compaction group (a row wider than its stride) is refused while the
    # call is planned: with no GPU, a call that reached its first launch would
    # report a CUDA error instead of APACK_EINVAL.
    import torch  # noqa: F401  (CPU tensors only: pointers are never dereferenced)
    s = make_seqs(ap)
    s.struct.modality = 0x1000
    n = ap.apack_workspace_size(s)
    ws = torch.zeros(n + 256, dtype=torch.uint8)
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + n]
    T, row = 65, 4 * 128 * 2
    kv = torch.zeros(2 * T * row, dtype=torch.uint8)
    out = torch.zeros(2 * T * row, dtype=torch.uint8)
    small = torch.zeros(4096, dtype=torch.int32)
    bad = ap.make_plane(small, out, 64, src_row_stride=32, dst_row_stride=64)
    counts = np.array([[5, 10], [2, 6]])
    with pytest.raises(ap.ApackError) as e:
        ap.apack_prune_step(s, 26, 28, small, kv, kv, T * row, None, 0, keep_count=counts, k_out=out, v_out=out,
                            kv_out_layer_stride=T * row, extra_planes=[bad], modality_out=small, keep_idx=small,
                            scores=small, ws=ws, stream=0)
    assert e.value.status == ap.APACK_EINVAL
    step = dict(layer=26, q=small, keep_count=counts, k_out=out, v_out=out, kv_out_layer_stride=T * row,
                modality_out=small, keep_idx=small, extra_planes=[bad])
    with pytest.raises(ap.ApackError) as e:
        ap.apack_prune_schedule(s, 28, kv, kv, T * row, None, 0, [step], scores=small, ws=ws, stream=0)
    assert e.value.status == ap.APACK_EINVAL
    # the same calls with a valid group get past planning and fail only at the device
    good = ap.make_plane(small, out, 64, src_row_stride=64, dst_row_stride=64)
    with pytest.raises(ap.ApackError) as e:
        ap.apack_prune_step(s, 26, 28, small, kv, kv, T * row, None, 0, keep_count=counts, k_out=out, v_out=out,
                            kv_out_layer_stride=T * row, extra_planes=[good], modality_out=small, keep_idx=small,
                            scores=small, ws=ws, stream=0)
    assert e.value.status == ap.APACK_ECUDA


def test_schedule_graph_holds_its_buffers_until_closed(ap):
    # a captured graph replays on the buffers it was captured on: the Python
    # object keeps them referenced, and drops them when it is closed
    import weakref

    class Buf:
        def data_ptr(self):
            return 0

    b = Buf()
    ref = weakref.ref(b)
    g = ap.ScheduleGraph(ctypes.c_void_p(None), [b])   # a null handle: close() calls nothing
    del b
    assert ref() is not None
    g.close()
    assert ref() is None
