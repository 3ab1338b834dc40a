"""Python binding of libapack, the GB300 (sm_103a) A-PACK inner-LLM prune step.

Argument marshalling only: every computation runs in the CUDA kernels of
``libapack.so`` behind the C ABI declared in ``include/apack.h``.  The
functions keep the C names (``apack_score``, ``apack_select``,
``apack_compact``, ``apack_prune_step``, ...).  Device buffers are passed as
torch CUDA tensors (their data pointers) and streams as torch streams;
PyTorch only provides memory and streams.

Importing this package loads the library and raises if it has not been
built (``__graft_entry__.build()`` or ``python -m paper_2608_08794_gb300._build``).
There is no fallback.
"""

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libapack.so")

APACK_OK, APACK_EINVAL, APACK_ECUDA, APACK_EWORKSPACE, APACK_ETIMEOUT, APACK_EDEVICE, APACK_EUNSUPPORTED = range(7)
APACK_MOD_OTHER, APACK_MOD_AUDIO, APACK_MOD_VISUAL = 0, 1, 2
APACK_SELECT_PER_MODALITY, APACK_SELECT_JOINT = 0, 1
APACK_SOFTMAX_MM, APACK_SOFTMAX_CAUSAL_ROW = 0, 1
APACK_HEAD_DIM = 128

EXPORTED = ("apack_workspace_size", "apack_keep_counts", "apack_score", "apack_select", "apack_compact",
            "apack_prune_step", "apack_device_error", "apack_launch_count", "apack_status_string",
            "apack_score_static", "apack_frame_alignment_workspace_size", "apack_frame_alignment",
            "apack_decode_workspace_size", "apack_decode_attention", "apack_prune_schedule",
            "apack_prune_schedule_graph", "apack_graph_launch", "apack_graph_destroy")


class ApackError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class apack_seqs(ctypes.Structure):
    _fields_ = [("num_seqs", ctypes.c_int32),
                ("cu_seqlens_h", ctypes.POINTER(ctypes.c_int32)),
                ("cu_qlens_h", ctypes.POINTER(ctypes.c_int32)),
                ("n_audio_h", ctypes.POINTER(ctypes.c_int32)),
                ("n_visual_h", ctypes.POINTER(ctypes.c_int32)),
                ("modality", ctypes.c_void_p),
                ("num_q_heads", ctypes.c_int32),
                ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32),
                ("softmax_domain", ctypes.c_int32),
                ("q_start_h", ctypes.POINTER(ctypes.c_int32))]


class apack_plane(ctypes.Structure):
    _fields_ = [("src", ctypes.c_void_p), ("dst", ctypes.c_void_p),
                ("src_plane_stride", ctypes.c_int64), ("dst_plane_stride", ctypes.c_int64),
                ("src_row_stride", ctypes.c_int64), ("dst_row_stride", ctypes.c_int64),
                ("row_bytes", ctypes.c_int64), ("num_planes", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class apack_step(ctypes.Structure):
    _fields_ = [("layer", ctypes.c_int32), ("q", ctypes.c_void_p),
                ("keep_count_h", ctypes.POINTER(ctypes.c_int32)), ("keep_ratio_h", ctypes.POINTER(ctypes.c_float)),
                ("k_out", ctypes.c_void_p), ("v_out", ctypes.c_void_p), ("kv_out_layer_stride", ctypes.c_int64),
                ("hidden_out", ctypes.c_void_p), ("extra_planes_h", ctypes.POINTER(apack_plane)),
                ("num_extra", ctypes.c_int32), ("modality_out", ctypes.c_void_p), ("keep_idx", ctypes.c_void_p),
                ("new_cu_seqlens_h", ctypes.POINTER(ctypes.c_int32)), ("new_cu_seqlens", ctypes.c_void_p)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"libapack.so is not built ({LIB_PATH}); run __graft_entry__.build()")
    lib = ctypes.CDLL(LIB_PATH)
    P, I32, I64, SZ, VP = ctypes.POINTER, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_void_p
    PI32 = P(I32)
    lib.apack_workspace_size.argtypes = [P(apack_seqs), P(SZ)]
    lib.apack_keep_counts.argtypes = [P(apack_seqs), P(ctypes.c_float), I32, PI32, PI32]
    lib.apack_score.argtypes = [P(apack_seqs), VP, VP, I64, VP, VP, SZ, VP]
    lib.apack_select.argtypes = [P(apack_seqs), VP, P(ctypes.c_float), PI32, I32, VP, VP, VP, VP, VP, SZ, VP]
    lib.apack_compact.argtypes = [VP, I64, P(apack_plane), I32, VP, VP]
    lib.apack_prune_step.argtypes = [P(apack_seqs), I32, I32, VP, VP, VP, I64, VP, I64, P(ctypes.c_float), PI32,
                                     I32, VP, VP, I64, VP, P(apack_plane), I32, VP, VP, PI32, VP, VP, VP, SZ,
                                     P(VP), VP]
    lib.apack_device_error.argtypes = [VP, VP, PI32, I32]
    lib.apack_score_static.argtypes = [P(apack_seqs), VP, VP, I64, VP, VP, VP]
    lib.apack_frame_alignment_workspace_size.argtypes = [I32, I64, P(SZ)]
    lib.apack_frame_alignment.argtypes = [VP, VP, I32, I32, I32, I64, I32, ctypes.c_float, ctypes.c_float, VP, VP,
                                          VP, VP, VP, SZ, VP]
    lib.apack_decode_workspace_size.argtypes = [I32, PI32, I32, I32, P(SZ)]
    lib.apack_decode_attention.argtypes = [I32, PI32, VP, VP, VP, I64, I32, I32, VP, VP, SZ, VP]
    lib.apack_prune_schedule.argtypes = [P(apack_seqs), I32, VP, VP, I64, VP, I64, I32, P(apack_step), I32, VP, VP,
                                         SZ, P(VP), VP]
    lib.apack_prune_schedule_graph.argtypes = [P(apack_seqs), I32, VP, VP, I64, VP, I64, I32, P(apack_step), I32,
                                               VP, VP, SZ, P(VP)]
    lib.apack_graph_launch.argtypes = [VP, VP]
    lib.apack_graph_destroy.argtypes = [VP]
    lib.apack_launch_count.argtypes = []
    lib.apack_launch_count.restype = ctypes.c_uint64
    lib.apack_status_string.argtypes = [I32]
    lib.apack_status_string.restype = ctypes.c_char_p
    for name in EXPORTED:
        if name not in ("apack_launch_count", "apack_status_string"):
            getattr(lib, name).restype = I32
    return lib


_lib = _load()


def status_string(status):
    return _lib.apack_status_string(int(status)).decode()


def _check(status, where):
    if status != APACK_OK:
        raise ApackError(status, where)


def _ptr(t):
    """Device pointer of a torch tensor (or None -> NULL)."""
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


def _i32(a):
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


class Seqs:
    """A packed batch: host offsets and counts plus the device modality mask.

    Keeps the host arrays alive for as long as the ``apack_seqs`` struct is used."""

    def __init__(self, cu_seqlens, cu_qlens, n_audio, n_visual, modality, num_q_heads, num_kv_heads,
                 head_dim=APACK_HEAD_DIM, softmax_domain=0, q_start=None):
        self.cu_seqlens = _i32(cu_seqlens)
        self.cu_qlens = _i32(cu_qlens)
        self.n_audio = _i32(n_audio)
        self.n_visual = _i32(n_visual)
        self.q_start = None if q_start is None else _i32(q_start)
        self.modality = modality
        I32P = ctypes.POINTER(ctypes.c_int32)
        self.struct = apack_seqs(
            num_seqs=len(self.cu_seqlens) - 1,
            cu_seqlens_h=self.cu_seqlens.ctypes.data_as(I32P),
            cu_qlens_h=self.cu_qlens.ctypes.data_as(I32P),
            n_audio_h=self.n_audio.ctypes.data_as(I32P),
            n_visual_h=self.n_visual.ctypes.data_as(I32P),
            modality=None if modality is None else modality.data_ptr(),
            num_q_heads=num_q_heads, num_kv_heads=num_kv_heads, head_dim=head_dim,
            softmax_domain=int(softmax_domain),
            q_start_h=None if self.q_start is None else self.q_start.ctypes.data_as(I32P))
        self.softmax_domain = int(softmax_domain)

    @property
    def num_seqs(self):
        return len(self.cu_seqlens) - 1

    @property
    def total_tokens(self):
        return int(self.cu_seqlens[-1])

    def ref(self):
        return ctypes.byref(self.struct)


def apack_workspace_size(seqs):
    n = ctypes.c_size_t(0)
    _check(_lib.apack_workspace_size(seqs.ref(), ctypes.byref(n)), "apack_workspace_size")
    return n.value


def apack_keep_counts(seqs, keep_ratio, select_mode=APACK_SELECT_PER_MODALITY):
    """Keep counts [B, 2] and new offsets [B+1] (host numpy) from keep ratios [B, 2]."""
    r = np.ascontiguousarray(np.asarray(keep_ratio, dtype=np.float32).reshape(seqs.num_seqs, 2))
    k = np.zeros((seqs.num_seqs, 2), np.int32)
    cu = np.zeros(seqs.num_seqs + 1, np.int32)
    I32P = ctypes.POINTER(ctypes.c_int32)
    _check(_lib.apack_keep_counts(seqs.ref(), r.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), select_mode,
                                  k.ctypes.data_as(I32P), cu.ctypes.data_as(I32P)), "apack_keep_counts")
    return k, cu


def apack_score(seqs, q, k, k_token_stride, scores, ws, stream=None):
    _check(_lib.apack_score(seqs.ref(), _ptr(q), _ptr(k), int(k_token_stride), _ptr(scores), _ptr(ws),
                            ws.numel() * ws.element_size(), _stream(stream)), "apack_score")


def apack_select(seqs, scores, keep_count, keep_idx, ws, select_mode=APACK_SELECT_PER_MODALITY,
                 modality_out=None, dst_of_src=None, new_cu_seqlens=None, stream=None, keep_ratio=None):
    """keep_count: [B, 2] counts, or None with keep_ratio [B, 2] (ratios 1-P of Eq. inner)."""
    kc = None if keep_count is None else _i32(keep_count).reshape(-1)
    kr = None if keep_ratio is None else np.ascontiguousarray(np.asarray(keep_ratio, np.float32).reshape(-1))
    _check(_lib.apack_select(seqs.ref(), _ptr(scores),
                             None if kr is None else kr.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                             None if kc is None else kc.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                             select_mode, _ptr(keep_idx), _ptr(modality_out), _ptr(dst_of_src),
                             _ptr(new_cu_seqlens), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "apack_select")


def make_plane(src, dst, row_bytes, num_planes=1, src_plane_stride=0, dst_plane_stride=0, src_row_stride=None,
               dst_row_stride=None):
    """Descriptor of a group of per-token planes (byte strides)."""
    return apack_plane(src=src.data_ptr(), dst=dst.data_ptr(), src_plane_stride=src_plane_stride,
                       dst_plane_stride=dst_plane_stride,
                       src_row_stride=row_bytes if src_row_stride is None else src_row_stride,
                       dst_row_stride=row_bytes if dst_row_stride is None else dst_row_stride,
                       row_bytes=row_bytes, num_planes=num_planes, reserved=0)


def apack_compact(keep_idx, n_out, planes, ws=None, stream=None):
    arr = (apack_plane * max(1, len(planes)))(*planes)
    _check(_lib.apack_compact(_ptr(keep_idx), int(n_out), arr, len(planes), _ptr(ws), _stream(stream)),
           "apack_compact")


def apack_prune_step(seqs, layer, num_layers, q, k_cache, v_cache, kv_layer_stride, hidden, hidden_dim,
                     keep_ratio=None, keep_count=None, select_mode=APACK_SELECT_PER_MODALITY, k_out=None,
                     v_out=None, kv_out_layer_stride=0, hidden_out=None, extra_planes=(), modality_out=None,
                     keep_idx=None, new_cu_seqlens=None, scores=None, ws=None, stage_events=None, stream=None):
    """One pruning step; returns the new packed offsets (host numpy [B+1])."""
    B = seqs.num_seqs
    I32P = ctypes.POINTER(ctypes.c_int32)
    ratio = None
    if keep_ratio is not None:
        ratio = np.ascontiguousarray(np.asarray(keep_ratio, dtype=np.float32).reshape(B, 2))
    kc = None if keep_count is None else _i32(keep_count).reshape(-1)
    new_cu = np.zeros(B + 1, np.int32)
    arr = (apack_plane * max(1, len(extra_planes)))(*extra_planes)
    ev = None
    if stage_events is not None:
        handles = [e.cuda_event if hasattr(e, "cuda_event") else e for e in stage_events]
        if len(handles) != 4 or not all(handles):
            raise ValueError("stage_events: four created CUDA events (record a torch event once to create it)")
        ev = (ctypes.c_void_p * 4)(*handles)
    st = _lib.apack_prune_step(
        seqs.ref(), int(layer), int(num_layers), _ptr(q), _ptr(k_cache), _ptr(v_cache), int(kv_layer_stride),
        _ptr(hidden), int(hidden_dim),
        None if ratio is None else ratio.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
        None if kc is None else kc.ctypes.data_as(I32P), select_mode, _ptr(k_out), _ptr(v_out),
        int(kv_out_layer_stride), _ptr(hidden_out), arr, len(extra_planes), _ptr(modality_out), _ptr(keep_idx),
        new_cu.ctypes.data_as(I32P), _ptr(new_cu_seqlens), _ptr(scores), _ptr(ws),
        0 if ws is None else ws.numel() * ws.element_size(), ev, _stream(stream))
    _check(st, "apack_prune_step")
    return new_cu


def _event_handles(events, n, what):
    if events is None:
        return None
    handles = [0 if e is None else (e.cuda_event if hasattr(e, "cuda_event") else e) for e in events]
    if len(handles) != n:
        raise ValueError(f"{what}: {n} events expected")
    return (ctypes.c_void_p * n)(*handles)


def apack_prune_schedule(seqs, num_layers, k_cache, v_cache, kv_layer_stride, hidden, hidden_dim, steps,
                         select_mode=APACK_SELECT_PER_MODALITY, scores=None, ws=None, stage_events=None, stream=None,
                         capture=False):
    """A whole progressive schedule (one apack_prune_step per entry of `steps`, each
    reading the previous step's outputs).  steps: dicts with layer, q, keep_count or
    keep_ratio, k_out, v_out, kv_out_layer_stride, hidden_out, modality_out, keep_idx
    and optionally new_cu_seqlens (device) and extra_planes.  stage_events: None or
    4 * len(steps) created events.  Returns the new host offsets of every step."""
    B = seqs.num_seqs
    n = len(steps)
    I32P = ctypes.POINTER(ctypes.c_int32)
    keep = []                           # host arrays referenced by the call
    arr = (apack_step * n)()
    new_cus = []
    for i, d in enumerate(steps):
        st = arr[i]
        st.layer = int(d["layer"])
        st.q = _ptr(d["q"])
        if d.get("keep_count") is not None:
            kc = _i32(d["keep_count"]).reshape(-1)
            keep.append(kc)
            st.keep_count_h = kc.ctypes.data_as(I32P)
        else:
            r = np.ascontiguousarray(np.asarray(d["keep_ratio"], dtype=np.float32).reshape(B, 2))
            keep.append(r)
            st.keep_ratio_h = r.ctypes.data_as(ctypes.POINTER(ctypes.c_float))
        st.k_out, st.v_out = _ptr(d["k_out"]), _ptr(d["v_out"])
        st.kv_out_layer_stride = int(d["kv_out_layer_stride"])
        st.hidden_out = _ptr(d.get("hidden_out"))
        extra = d.get("extra_planes", ())
        if extra:
            ep = (apack_plane * len(extra))(*extra)
            keep.append(ep)
            st.extra_planes_h = ctypes.cast(ep, ctypes.POINTER(apack_plane))
        st.num_extra = len(extra)
        st.modality_out = _ptr(d["modality_out"])
        st.keep_idx = _ptr(d["keep_idx"])
        cu = np.zeros(B + 1, np.int32)
        new_cus.append(cu)
        st.new_cu_seqlens_h = cu.ctypes.data_as(I32P)
        st.new_cu_seqlens = _ptr(d.get("new_cu_seqlens"))
    head = (seqs.ref(), int(num_layers), _ptr(k_cache), _ptr(v_cache), int(kv_layer_stride), _ptr(hidden),
            int(hidden_dim), int(select_mode), arr, n, _ptr(scores), _ptr(ws),
            0 if ws is None else ws.numel() * ws.element_size())
    if capture:
        g = ctypes.c_void_p()
        _check(_lib.apack_prune_schedule_graph(*head, ctypes.byref(g)), "apack_prune_schedule_graph")
        # the graph replays on these device buffers: keep them alive with it
        buffers = [t for t in (k_cache, v_cache, hidden, scores, ws, seqs.modality) if t is not None]
        for d in steps:
            buffers += [v for v in d.values() if hasattr(v, "data_ptr")]
        return new_cus, ScheduleGraph(g, buffers)
    stage = _event_handles(stage_events, 4 * n, "stage_events")
    _check(_lib.apack_prune_schedule(*head, stage, _stream(stream)), "apack_prune_schedule")
    return new_cus


class ScheduleGraph:
    """An executable CUDA graph of one schedule (apack_prune_schedule_graph);
    launch() replays it, the graph is freed with the object.  The graph reads
    and writes the device buffers it was captured on, so the object holds
    references to them (inputs, outputs, scores, workspace) until it is closed."""

    def __init__(self, handle, buffers=()):
        self._h = handle
        self._buffers = list(buffers)

    def launch(self, stream=None):
        _check(_lib.apack_graph_launch(self._h, _stream(stream)), "apack_graph_launch")

    def close(self):
        if self._h is not None and self._h.value:
            _check(_lib.apack_graph_destroy(self._h), "apack_graph_destroy")
        self._h = None
        self._buffers = []

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def apack_prune_schedule_graph(seqs, num_layers, k_cache, v_cache, kv_layer_stride, hidden, hidden_dim, steps,
                               select_mode=APACK_SELECT_PER_MODALITY, scores=None, ws=None):
    """Captures the schedule of apack_prune_schedule (same arguments) into a CUDA
    graph.  Returns (new host offsets of every step, ScheduleGraph)."""
    return apack_prune_schedule(seqs, num_layers, k_cache, v_cache, kv_layer_stride, hidden, hidden_dim, steps,
                                select_mode=select_mode, scores=scores, ws=ws, capture=True)


def apack_score_static(seqs, q, k, k_token_stride, scores, device_error_out=None, stream=None):
    """apack_score without a workspace, for callers that cannot allocate device
    memory (the library's fixed 8 MiB scratch array is used instead)."""
    _check(_lib.apack_score_static(seqs.ref(), _ptr(q), _ptr(k), int(k_token_stride), _ptr(scores),
                                   _ptr(device_error_out), _stream(stream)), "apack_score_static")


def apack_frame_alignment_workspace_size(n_frames, dim):
    n = ctypes.c_size_t(0)
    _check(_lib.apack_frame_alignment_workspace_size(int(n_frames), int(dim), ctypes.byref(n)),
           "apack_frame_alignment_workspace_size")
    return n.value


def apack_frame_alignment(visual, audio, n_frames, tokens_per_frame, n_audio, dim, c_out, s_out, ws, window=3,
                          tau=0.78, beta=0.90, dnorm_out=None, cbar_out=None, stream=None):
    """Pre-LLM windowed CKA c_f and gated score s_f per frame (Sec. 3.1)."""
    _check(_lib.apack_frame_alignment(_ptr(visual), _ptr(audio), int(n_frames), int(tokens_per_frame), int(n_audio),
                                      int(dim), int(window), float(tau), float(beta), _ptr(c_out), _ptr(s_out),
                                      _ptr(dnorm_out), _ptr(cbar_out), _ptr(ws), ws.numel() * ws.element_size(),
                                      _stream(stream)), "apack_frame_alignment")


def apack_decode_workspace_size(cu_seqlens, num_q_heads, num_kv_heads):
    cu = _i32(cu_seqlens)
    n = ctypes.c_size_t(0)
    _check(_lib.apack_decode_workspace_size(len(cu) - 1, cu.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), int(num_q_heads),
                                            int(num_kv_heads), ctypes.byref(n)), "apack_decode_workspace_size")
    return n.value


def apack_decode_attention(cu_seqlens, q, k, v, kv_token_stride, num_q_heads, num_kv_heads, out, ws, stream=None):
    """Attention of one decode token per sequence over its KV cache (Sec. 3.2)."""
    cu = _i32(cu_seqlens)
    _check(_lib.apack_decode_attention(len(cu) - 1, cu.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), _ptr(q), _ptr(k), _ptr(v),
                                       int(kv_token_stride), int(num_q_heads), int(num_kv_heads), _ptr(out),
                                       _ptr(ws), ws.numel() * ws.element_size(), _stream(stream)),
           "apack_decode_attention")


def apack_device_error(ws, stream=None, clear=True):
    code = ctypes.c_int32(0)
    _check(_lib.apack_device_error(_ptr(ws), _stream(stream), ctypes.byref(code), 1 if clear else 0),
           "apack_device_error")
    return code.value


def apack_launch_count():
    return int(_lib.apack_launch_count())


def library_path():
    return LIB_PATH
