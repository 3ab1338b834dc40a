"""Device twin of the generator: fills torch CUDA tensors with the same bf16
bits that ``synth.gen.normal_bf16_bits`` produces on the host."""

import ctypes
import os

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libsynth_fill.so")
_lib = None


def _load():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is not built; run __graft_entry__.build()")
        lib = ctypes.CDLL(LIB_PATH)
        lib.synth_fill_normal_bf16.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint64,
                                               ctypes.c_uint64, ctypes.c_void_p]
        lib.synth_fill_normal_bf16.restype = ctypes.c_int
        _lib = lib
    return _lib


def fill_normal_bf16(t, seed, tid, start=0, stream=None):
    """Fill a contiguous 16-bit CUDA tensor with draws start.. of stream (seed, tid)."""
    import torch
    assert t.is_cuda and t.element_size() == 2 and t.is_contiguous()
    if stream is None:
        stream = torch.cuda.current_stream()
    rc = _load().synth_fill_normal_bf16(ctypes.c_void_p(t.data_ptr()), t.numel(), seed, tid, start,
                                        ctypes.c_void_p(stream.cuda_stream))
    if rc != 0:
        raise RuntimeError("synth_fill_normal_bf16 failed")


def fill_progressive_inputs(pp, wl):
    """Fills the input buffers of a ``ProgressivePrune`` for workload ``wl``:
    K/V of layers [l_0, L) drawn on the device, plants written into the K
    slabs of every pruning layer, Q of every pruning layer, hidden states and
    the modality mask.  Returns the host Q arrays (uint16) per step."""
    import numpy as np
    import torch
    from .gen import TID_K, TID_V, TID_HIDDEN
    from .inputs import query_rows, plant_patch
    l0 = wl.prune_layers[0]
    for j in range(pp.k_in.shape[0]):
        fill_normal_bf16(pp.k_in[j], wl.seed, TID_K + l0 + j)
        fill_normal_bf16(pp.v_in[j], wl.seed, TID_V + l0 + j)
    if getattr(pp, "slice_below", False):
        for j in range(pp.k_low_in.shape[0]):
            fill_normal_bf16(pp.k_low_in[j], wl.seed, TID_K + j)
            fill_normal_bf16(pp.v_low_in[j], wl.seed, TID_V + j)
    if pp.hidden_in is not None:
        fill_normal_bf16(pp.hidden_in, wl.seed, TID_HIDDEN)
    pp.modality_in.copy_(torch.from_numpy(wl.modality()))
    qs = []
    for i, layer in enumerate(wl.prune_layers):
        q = query_rows(wl, layer)
        qs.append(q)
        pp.q[i].copy_(torch.from_numpy(q.view(np.int16)).view(torch.bfloat16))
        tok, rows = plant_patch(wl, layer, q)
        if tok.size:
            idx = torch.from_numpy(tok).to(pp.k_in.device)
            pp.k_in[layer - l0].index_copy_(0, idx, torch.from_numpy(rows.view(np.int16)).view(torch.bfloat16)
                                            .to(pp.k_in.device))
    torch.cuda.synchronize()
    return qs
