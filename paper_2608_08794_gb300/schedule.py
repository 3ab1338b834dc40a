"""Host-side driver of a progressive pruning schedule (Algorithm 1, the loop
over pruning layers l >= L_mid; Sec. 3.2: pruning repeats at later layers on
the already shortened sequence).

Step i prunes at layer l_i and compacts the K/V slabs of layers [l_i, L)
plus the hidden states; step i+1 reads its layer's keys from slab
(l_{i+1} - l_i) of step i's output.  Two output buffers alternate
(ping-pong), so the input cache of step 0 is never written and the schedule
can be replayed on the same inputs.  ``run_step`` calls ``apack_prune_step``
for one step; ``run`` hands the whole schedule to ``apack_prune_schedule``.

Only buffer management and argument marshalling happen here.
"""

import numpy as np
import torch

from . import (Seqs, apack_plane, apack_prune_step, apack_prune_schedule, apack_prune_schedule_graph,
               apack_workspace_size, apack_keep_counts, apack_score, apack_select, apack_compact, make_plane,
               APACK_HEAD_DIM, APACK_SELECT_PER_MODALITY, APACK_SELECT_JOINT)


def _wait(waiter, producer):
    """Orders `waiter` after the work queued so far on `producer` (torch streams or None)."""
    w = waiter if waiter is not None else torch.cuda.current_stream()
    p = producer if producer is not None else torch.cuda.current_stream()
    ev = torch.cuda.Event()
    ev.record(p)
    w.wait_event(ev)


def _plane(src, dst, src_plane_stride, dst_plane_stride, row_bytes, num_planes):
    return apack_plane(src=src, dst=dst, src_plane_stride=src_plane_stride, dst_plane_stride=dst_plane_stride,
                       src_row_stride=row_bytes, dst_row_stride=row_bytes, row_bytes=row_bytes,
                       num_planes=num_planes)


def schedule_keep_counts(cu_seqlens, cu_qlens, n_audio, n_visual, num_q_heads, num_kv_heads, modality,
                         steps, cumulative_ratios=None, joint_step_keep=None):
    """Keep counts [B, 2] of every step of a schedule, from the library's rule
    (ceil((1-P)|S|) of Eq. inner, apack_keep_counts), and the selection mode.

    cumulative_ratios[i][b] = (audio, visual) keep ratios of step i, applied to
    the counts entering step 0 (per-modality selection); or joint_step_keep =
    the fraction of the current |S| each step keeps (the paper's joint form)."""
    na = np.asarray(n_audio, np.int32)
    nv = np.asarray(n_visual, np.int32)
    if joint_step_keep is None:
        s0 = Seqs(cu_seqlens, cu_qlens, na, nv, modality, num_q_heads, num_kv_heads)
        counts = [apack_keep_counts(s0, np.asarray(r, np.float32))[0] for r in cumulative_ratios]
        return counts, APACK_SELECT_PER_MODALITY
    counts, n = [], na + nv
    for _ in range(steps):
        s = Seqs(cu_seqlens, cu_qlens, n, np.zeros_like(n), modality, num_q_heads, num_kv_heads)
        k, _ = apack_keep_counts(s, np.full((len(n), 2), joint_step_keep, np.float32), APACK_SELECT_JOINT)
        counts.append(k)
        n = k[:, 0].copy()
    return counts, APACK_SELECT_JOINT


class ProgressivePrune:
    def __init__(self, cu_seqlens, cu_qlens, n_audio, n_visual, num_q_heads, num_kv_heads, num_layers, hidden_dim,
                 prune_layers, keep_counts, device="cuda", select_mode=APACK_SELECT_PER_MODALITY,
                 with_hidden=True, slice_below=False, softmax_domain=0, in_place=False):
        """keep_counts[i]: int array [B, 2] of the tokens each segment keeps after step i.

        slice_below: also compact, at every step, the K/V of the layers below its
        pruning layer, so that after the schedule every layer's cache holds only the
        kept tokens (for decoding).  The caches of layers [0, l_0) are then inputs
        too (``k_low_in`` / ``v_low_in``); ``output_low_kv`` gives layers [0, l_i).

        in_place: every step compacts within the input buffers (k_in, v_in, hidden_in keep their
        slab stride; step i's result is the first t_out_i rows of slabs l_i - l_0 ..), so no
        output caches are allocated: a third of the memory, at the in-place gather's speed.
        softmax_domain: APACK_SOFTMAX_MM (default) or APACK_SOFTMAX_CAUSAL_ROW."""
        self.dev = torch.device(device)
        self.softmax_domain = int(softmax_domain)
        self.cu0 = np.asarray(cu_seqlens, np.int32)
        self.cuq = np.asarray(cu_qlens, np.int32)
        self.na0 = np.asarray(n_audio, np.int32)
        self.nv0 = np.asarray(n_visual, np.int32)
        self.hq, self.hkv, self.L, self.H = num_q_heads, num_kv_heads, num_layers, hidden_dim
        self.layers = list(prune_layers)
        self.counts = [np.asarray(k, np.int32).reshape(-1, 2) for k in keep_counts]
        self.mode = select_mode
        self.row = num_kv_heads * APACK_HEAD_DIM * 2
        self.T0 = int(self.cu0[-1])
        self.B = len(self.cu0) - 1
        other = np.diff(self.cu0) - self.na0 - self.nv0
        self.t_out = [int((other + k[:, 0] + k[:, 1]).sum()) for k in self.counts]
        dev, T0, Lc0 = self.dev, self.T0, num_layers - self.layers[0]
        # inputs (filled by the caller): K/V of layers [l_0, L), hidden, modality, Q per step
        self.k_in = torch.empty((Lc0, T0, num_kv_heads, APACK_HEAD_DIM), dtype=torch.bfloat16, device=dev)
        self.v_in = torch.empty_like(self.k_in)
        self.hidden_in = torch.empty((T0, hidden_dim), dtype=torch.bfloat16, device=dev) if with_hidden else None
        self.modality_in = torch.empty(T0, dtype=torch.uint8, device=dev)
        nq = int(self.cuq[-1])
        self.q = [torch.empty((nq, num_q_heads, APACK_HEAD_DIM), dtype=torch.bfloat16, device=dev)
                  for _ in self.layers]
        # outputs, sized for the largest step (ping-pong), or the inputs themselves (in place: every
        # step compacts its slabs of k_in / v_in and hidden_in within their own rows)
        t1 = self.t_out[0]
        self.in_place = bool(in_place)
        if self.in_place and slice_below:
            raise ValueError("in_place and slice_below cannot be combined")
        if self.in_place:
            self.k_out = self.v_out = self.h_out = None
        else:
            self.k_out = [torch.empty(Lc0 * t1 * self.row // 2, dtype=torch.bfloat16, device=dev) for _ in range(2)]
            self.v_out = [torch.empty_like(self.k_out[0]) for _ in range(2)]
            self.h_out = [torch.empty((t1, hidden_dim), dtype=torch.bfloat16, device=dev) if with_hidden else None
                          for _ in range(2)]
        self.mod_out = [torch.empty(t1, dtype=torch.uint8, device=dev) for _ in range(2)]
        self.slice_below = slice_below
        if slice_below:
            l0, l_last = self.layers[0], self.layers[-1]
            self.k_low_in = torch.empty((l0, T0, num_kv_heads, APACK_HEAD_DIM), dtype=torch.bfloat16, device=dev)
            self.v_low_in = torch.empty_like(self.k_low_in)
            self.k_low = [torch.empty(max(1, l_last * t1 * self.row // 2), dtype=torch.bfloat16, device=dev)
                          for _ in range(2)]
            self.v_low = [torch.empty_like(self.k_low[0]) for _ in range(2)]
        self.keep_idx = [torch.empty(max(1, t), dtype=torch.int32, device=dev) for t in self.t_out]
        self.scores = torch.empty(max(1, T0), dtype=torch.float32, device=dev)
        self._seqs = []
        ws_bytes = 0
        for i in range(len(self.layers)):
            s = self._step_seqs(i)
            ws_bytes = max(ws_bytes, apack_workspace_size(s))
        self.ws = torch.zeros(ws_bytes + 256, dtype=torch.uint8, device=dev)
        off = (-self.ws.data_ptr()) % 256
        self.ws = self.ws[off:off + ws_bytes]
        self.new_cu = []

    def _step_seqs(self, i):
        if i < len(self._seqs):
            return self._seqs[i]
        if i == 0:
            cu, na, nv, mod = self.cu0, self.na0, self.nv0, self.modality_in
        else:
            other = np.diff(self.cu0) - self.na0 - self.nv0
            k = self.counts[i - 1]
            cu = np.concatenate([[0], np.cumsum(other + k[:, 0] + k[:, 1])]).astype(np.int32)
            na, nv = k[:, 0], k[:, 1]
            mod = self.mod_out[(i - 1) % 2]
        s = Seqs(cu, self.cuq, na, nv, mod, self.hq, self.hkv, softmax_domain=self.softmax_domain)
        self._seqs.append(s)
        return s

    def step_args(self, i):
        """(seqs, k_in, v_in, in_layer_stride, hidden_in) entering step i; K/V as flat bf16 views."""
        if i == 0:
            return (self._step_seqs(0), self.k_in.view(-1), self.v_in.view(-1), self.T0 * self.row, self.hidden_in)
        k_prev, v_prev, stride = self.step_outputs(i - 1)
        off = (self.layers[i] - self.layers[i - 1]) * stride // 2     # bf16 elements
        return (self._step_seqs(i), k_prev[off:], v_prev[off:], stride, self.step_hidden_out(i - 1))

    def step_outputs(self, i):
        """(k_out, v_out, slab stride in bytes) that step i writes: flat bf16 views."""
        if self.in_place:
            off = (self.layers[i] - self.layers[0]) * self.T0 * self.row // 2
            return self.k_in.view(-1)[off:], self.v_in.view(-1)[off:], self.T0 * self.row
        o = i % 2
        return self.k_out[o], self.v_out[o], self.t_out[i] * self.row

    def step_hidden_out(self, i):
        return self.hidden_in if self.in_place else self.h_out[i % 2]

    def _schedule_steps(self):
        steps = []
        for i in range(len(self.layers)):
            o = i % 2
            k_out, v_out, stride = self.step_outputs(i)
            steps.append(dict(layer=self.layers[i], q=self.q[i], keep_count=self.counts[i], k_out=k_out,
                              v_out=v_out, kv_out_layer_stride=stride,
                              hidden_out=self.step_hidden_out(i), modality_out=self.mod_out[o], keep_idx=self.keep_idx[i],
                              extra_planes=self._below_planes(i)))
        return steps

    def run(self, events=None, stream=None):
        """Runs every step through apack_prune_schedule.  events: None or 4 CUDA
        events per step (before scoring, after scoring, after selection, after
        compaction)."""
        flat = None
        if events is not None:
            flat = [e for per_step in events for e in per_step]
        self.new_cu = apack_prune_schedule(
            self._step_seqs(0), self.L, self.k_in.view(-1), self.v_in.view(-1), self.T0 * self.row,
            self.hidden_in, self.H, self._schedule_steps(), select_mode=self.mode, scores=self.scores, ws=self.ws,
            stage_events=flat, stream=stream)

    def capture(self):
        """The schedule of run() as a CUDA graph (apack_prune_schedule_graph):
        graph.launch(stream) replays every launch with these buffers."""
        self.new_cu, graph = apack_prune_schedule_graph(
            self._step_seqs(0), self.L, self.k_in.view(-1), self.v_in.view(-1), self.T0 * self.row,
            self.hidden_in, self.H, self._schedule_steps(), select_mode=self.mode, scores=self.scores, ws=self.ws)
        return graph

    def run_first_step_from_host(self, k_host, v_host, hidden_host=None, stream=None):
        """Step 0 with the K/V caches of layers [l_0, L) (and the hidden states) in pinned host
        memory, laid out like k_in / v_in / hidden_in.  Only the scored layer's keys must be on
        the device: the caller copies slab 0 of k_in.  Scoring and selection run on the device;
        the compaction reads only the kept rows over the host link (apack_compact from a host
        source).  Leaves exactly what run_step(0) leaves; continue with run_step(1), ..."""
        self.select_first_step(stream=stream)
        self.compact_first_step_from_host(k_host, v_host, hidden_host, stream=stream)

    def select_first_step(self, stream=None):
        """Scoring and selection of step 0 on the device (slab 0 of k_in holds the scored keys):
        the first half of run_first_step_from_host."""
        if self.slice_below or self.in_place:
            raise ValueError("run_first_step_from_host: slice_below and in_place are not supported")
        seqs = self._step_seqs(0)
        apack_score(seqs, self.q[0], self.k_in.view(-1), self.row, self.scores, self.ws, stream=stream)
        apack_select(seqs, self.scores, self.counts[0], self.keep_idx[0], self.ws, select_mode=self.mode,
                     modality_out=self.mod_out[0], stream=stream)

    def compact_first_step_from_host(self, k_host, v_host, hidden_host=None, stream=None):
        """The compaction of step 0 from host-resident caches (after select_first_step on the
        stream order): only the kept rows cross the host link."""
        t_out, lc = self.t_out[0], self.L - self.layers[0]
        new_cu = np.zeros(self.B + 1, np.int32)
        planes = [make_plane(k_host, self.k_out[0], self.row, lc, self.T0 * self.row, t_out * self.row),
                  make_plane(v_host, self.v_out[0], self.row, lc, self.T0 * self.row, t_out * self.row)]
        if hidden_host is not None and self.h_out[0] is not None:
            planes.append(make_plane(hidden_host, self.h_out[0], self.H * 2, 1))
        apack_compact(self.keep_idx[0], t_out, planes, ws=self.ws, stream=stream)
        other = np.diff(self.cu0) - self.na0 - self.nv0
        k = self.counts[0]
        new_cu[1:] = np.cumsum(other + k[:, 0] + k[:, 1])
        if len(self.new_cu) != len(self.layers):
            self.new_cu = [None] * len(self.layers)
        self.new_cu[0] = new_cu

    def _final_buffers(self):
        """Buffers of run_from_host, allocated on first use: every layer's cache at the level it
        ends at (k_fin[i] / v_fin[i]: layers [l_i, l_(i+1)) at t_out_i rows), the scored keys of
        each later step at the level that step reads (k_score[i]: layer l_i at t_out_(i-1) rows)
        and the composed row indices into the step-0 input (comp[i], i >= 1)."""
        if getattr(self, "k_fin", None) is not None:
            return
        n = len(self.layers)
        ends = self.layers[1:] + [self.L]
        self.fin_layers = [e - l for l, e in zip(self.layers, ends)]
        self.k_fin = [torch.empty((c, max(1, t), self.hkv, APACK_HEAD_DIM), dtype=torch.bfloat16, device=self.dev)
                      for c, t in zip(self.fin_layers, self.t_out)]
        self.v_fin = [torch.empty_like(k) for k in self.k_fin]
        self.k_score = [None] + [torch.empty((max(1, self.t_out[i - 1]), self.hkv, APACK_HEAD_DIM),
                                             dtype=torch.bfloat16, device=self.dev) for i in range(1, n)]
        self.comp = [None] + [torch.empty(max(1, t), dtype=torch.int32, device=self.dev) for t in self.t_out[1:]]
        self.gather_done = [torch.cuda.Event() for _ in range(n)]

    def run_from_host(self, k_host, v_host, hidden_host=None, stream=None, gather_stream=None):
        """The whole schedule with the K/V caches of layers [l_0, L) and the hidden states in pinned
        host memory (laid out like k_in / v_in / hidden_in; the caller copies the scored keys,
        slab 0 of k_in, to the device).  Every layer's rows cross the host link once, at the level
        that layer ends at: step i gathers, at the composed indices of steps 0..i, the K and V of
        layers [l_i, l_(i+1)) and the keys that step i+1 scores (layer l_(i+1)); the last step
        also gathers the hidden states.  Only the scored keys of step i (already on the device)
        are compacted on the device.
        Scoring and selection are those of run_step, so keep_idx, scores and the caches equal the
        per-step schedule's bit for bit; the result is every layer's final cache (final_kv),
        output_hidden(last) and keep_idx.  gather_stream: None, or a stream for the host-link
        gathers (ordered against `stream` with events).  The sources may also be device buffers
        (k_in, v_in, hidden_in themselves): the same schedule then writes every layer once on the
        device, where the per-step schedule compacts layers [l_i, L) at every step."""
        for i in range(len(self.layers)):
            self.host_step(i, k_host, v_host, hidden_host, stream=stream, gather_stream=gather_stream)

    def host_step(self, i, k_host, v_host, hidden_host=None, stream=None, gather_stream=None):
        """Step i of run_from_host (steps run in order; step 0 needs the scored keys in slab 0 of
        k_in).  After the last step, `stream` is ordered after every gather."""
        if self.slice_below or self.in_place:
            raise ValueError("run_from_host: slice_below and in_place are not supported")
        self._final_buffers()
        n, row, T0 = len(self.layers), self.row, self.T0
        gs = gather_stream if gather_stream is not None else stream
        kh, vh = k_host.data_ptr(), v_host.data_ptr()
        if len(self.new_cu) != n:
            self.new_cu = [None] * n
        other = np.diff(self.cu0) - self.na0 - self.nv0
        seqs = self._step_seqs(i)
        t = self.t_out[i]
        k_sc = self.k_in.view(-1) if i == 0 else self.k_score[i]
        if i > 0 and gs is not stream:
            # the scored keys came over the link in step i-1's gather; later gathers queued on gs
            # meanwhile (another schedule's) need not end
            (stream or torch.cuda.current_stream()).wait_event(self.gather_done[i - 1])
        apack_score(seqs, self.q[i], k_sc, row, self.scores, self.ws, stream=stream)
        apack_select(seqs, self.scores, self.counts[i], self.keep_idx[i], self.ws, select_mode=self.mode,
                     modality_out=self.mod_out[i % 2], stream=stream)
        if i > 0:                              # rows of the step-0 input that step i keeps
            prev = self.keep_idx[0] if i == 1 else self.comp[i - 1]
            apack_compact(self.keep_idx[i], t, [make_plane(prev, self.comp[i], 4, 1)], stream=stream)
        comp = self.keep_idx[0] if i == 0 else self.comp[i]
        # host-link gathers of this step, at the composed indices
        l0, li = self.layers[0], self.layers[i]
        c = self.fin_layers[i]
        kf, vf = self.k_fin[i].data_ptr(), self.v_fin[i].data_ptr()
        planes = [_plane(vh + (li - l0) * T0 * row, vf, T0 * row, t * row, row, c)]
        k_first = 0 if i == 0 else 1           # layer l_i's keys of a later step come from the device
        if c > k_first:
            planes.append(_plane(kh + (li - l0 + k_first) * T0 * row, kf + k_first * t * row, T0 * row,
                                 t * row, row, c - k_first))
        if i + 1 < n:
            planes.append(_plane(kh + (self.layers[i + 1] - l0) * T0 * row, self.k_score[i + 1].data_ptr(),
                                 T0 * row, t * row, row, 1))
        if i + 1 == n and hidden_host is not None and self.h_out[0] is not None:
            # the hidden states cross once too, at the level they end at
            planes.append(make_plane(hidden_host, self.h_out[i % 2], self.H * 2, 1))
        if gs is not stream:
            _wait(gs, stream)
        apack_compact(comp, t, planes, ws=self.ws, stream=gs)
        if gs is not stream:
            self.gather_done[i].record(gs)
        if i > 0:                              # device-side: layer l_i's keys, scored above
            apack_compact(self.keep_idx[i], t, [_plane(self.k_score[i].data_ptr(), kf, 0, 0, row, 1)], ws=self.ws,
                          stream=stream)
        k = self.counts[i]
        cu = np.zeros(self.B + 1, np.int32)
        cu[1:] = np.cumsum(other + k[:, 0] + k[:, 1])
        self.new_cu[i] = cu
        if i + 1 == n and gs is not stream:
            (stream or torch.cuda.current_stream()).wait_event(self.gather_done[i])

    def final_kv(self, i):
        """run_from_host's caches of layers [l_i, l_(i+1)) (the last step: [l_i, L)) at their final
        level: [n_layers, t_out_i, Hkv, D] K and V."""
        t = self.t_out[i]
        return self.k_fin[i][:, :t], self.v_fin[i][:, :t]

    def run_steps(self, events=None, stream=None):
        """Runs every step with one apack_prune_step call each; events[i] = 4 CUDA
        events per step or None."""
        self.new_cu = [None] * len(self.layers)
        for i in range(len(self.layers)):
            self.run_step(i, None if events is None else events[i], stream)

    def run_step(self, i, events=None, stream=None):
        if len(self.new_cu) != len(self.layers):
            self.new_cu = [None] * len(self.layers)
        seqs, k, v, stride, h = self.step_args(i)
        o = i % 2
        k_out, v_out, out_stride = self.step_outputs(i)
        self.new_cu[i] = apack_prune_step(
            seqs, self.layers[i], self.L, self.q[i], k, v, stride, h, self.H, keep_count=self.counts[i],
            select_mode=self.mode, k_out=k_out, v_out=v_out, kv_out_layer_stride=out_stride,
            hidden_out=self.step_hidden_out(i), modality_out=self.mod_out[o], keep_idx=self.keep_idx[i],
            scores=self.scores, ws=self.ws, stage_events=events, stream=stream)
        return self.new_cu[i]

    def _below_planes(self, i):
        """Extra planes of step i when slicing below: layers [0, l_(i-1)) from the
        previous below-cache and layers [l_(i-1), l_i) from the previous step's main
        output (for step 0: layers [0, l_0) from the inputs), into layers [0, l_i)."""
        if not self.slice_below:
            return ()
        row, t = self.row, self.t_out[i]
        o = i % 2
        groups = []
        for src_in, out, low in ((self.k_low_in, self.k_out, self.k_low), (self.v_low_in, self.v_out, self.v_low)):
            dst = low[o].data_ptr()
            if i == 0:
                if self.layers[0] > 0:
                    groups.append(_plane(src_in.data_ptr(), dst, self.T0 * row, t * row, row, self.layers[0]))
                continue
            p, tp = (i - 1) % 2, self.t_out[i - 1]
            lp, li = self.layers[i - 1], self.layers[i]
            if lp > 0:
                groups.append(_plane(low[p].data_ptr(), dst, tp * row, t * row, row, lp))
            groups.append(_plane(out[p].data_ptr(), dst + lp * t * row, tp * row, t * row, row, li - lp))
        return groups

    def output_low_kv(self, i):
        """Views of step i's below-layer caches (slice_below): [l_i, t_out_i, Hkv, D]."""
        o = i % 2
        n = self.layers[i] * self.t_out[i] * self.row // 2
        shape = (self.layers[i], self.t_out[i], self.hkv, APACK_HEAD_DIM)
        return self.k_low[o][:n].view(shape), self.v_low[o][:n].view(shape)

    def output_kv(self, i):
        """Views of step i's compacted K and V: [L - l_i, t_out_i, Hkv, D] (in place: strided
        views into k_in / v_in, valid until a later step compacts them again)."""
        if self.in_place:
            s = self.layers[i] - self.layers[0]
            return self.k_in[s:, :self.t_out[i]], self.v_in[s:, :self.t_out[i]]
        o = i % 2
        n = (self.L - self.layers[i]) * self.t_out[i] * self.row // 2
        shape = (self.L - self.layers[i], self.t_out[i], self.hkv, APACK_HEAD_DIM)
        return self.k_out[o][:n].view(shape), self.v_out[o][:n].view(shape)

    def output_hidden(self, i):
        h = self.step_hidden_out(i)
        return None if h is None else h[:self.t_out[i]]

    def mm_tokens_per_step(self):
        """|S| entering each step (the unit of the throughput metric)."""
        out = [int(self.na0.sum() + self.nv0.sum())]
        for k in self.counts[:-1]:
            out.append(int(k.sum()))
        return out
