// schedule.cu -- a whole progressive pruning schedule in one call (Sec. 3.2: pruning
// repeated at later layers, each step retaining a fraction of the current tokens;
// Algorithm 1, the inner-LLM loop over layers).
//
// Step i scores and selects with layer l_i's keys, then compacts K/V of layers [l_i, L),
// the hidden states and any extra planes to the kept tokens; step i+1 reads step i's
// outputs.  All steps are planned and checked on the host before the first launch, then
// run in order on one stream: the outputs are those of one apack_prune_step per step.
#include <new>
#include <vector>

#include "internal.cuh"

namespace apack {
namespace {

struct StepPlan {
  std::vector<int32_t> cu, na, nv;     // sequences entering the step
  std::vector<int32_t> counts;         // [B][2] kept per (sequence, modality) or (|S|, 0) jointly
  apack_seqs seqs{};
  const void *k = nullptr, *v = nullptr, *hidden = nullptr;
  int64_t kv_layer_stride = 0;
  std::vector<apack_plane> planes;     // the step's compaction groups
};

apack_plane plane(const void *src, void *dst, int64_t src_ps, int64_t dst_ps, int64_t row, int32_t n) {
  apack_plane p{};
  p.src = src;
  p.dst = dst;
  p.src_plane_stride = src_ps;
  p.dst_plane_stride = dst_ps;
  p.src_row_stride = row;
  p.dst_row_stride = row;
  p.row_bytes = row;
  p.num_planes = n;
  return p;
}

}  // namespace
}  // namespace apack

using namespace apack;

extern "C" {

apack_status apack_prune_schedule(const apack_seqs *seqs, int32_t num_layers, const void *k_cache,
                                  const void *v_cache, int64_t kv_layer_stride, const void *hidden,
                                  int64_t hidden_dim, int32_t select_mode, const apack_step *steps_h,
                                  int32_t num_steps, float *scores, void *ws, size_t ws_bytes,
                                  void *const *stage_events_h, void *stream) {
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (num_steps < 1 || !steps_h || !k_cache || !v_cache || !scores) return APACK_EINVAL;
  if (in_host_memory(k_cache)) return APACK_EINVAL;   // scored by TMA: device memory
  if (hidden && hidden_dim <= 0) return APACK_EINVAL;
  const int B = seqs->num_seqs;
  const int64_t row = static_cast<int64_t>(seqs->num_kv_heads) * APACK_HEAD_DIM * 2;

  // plan every step on the host first: nothing is launched unless all steps are valid
  DeviceError *err =
      ws ? reinterpret_cast<DeviceError *>(static_cast<uint8_t *>(ws) + workspace_layout(seqs).err_off) : nullptr;
  std::vector<StepPlan> plan(static_cast<size_t>(num_steps));
  for (int i = 0; i < num_steps; ++i) {
    const apack_step &sp = steps_h[i];
    StepPlan &p = plan[i];
    if (sp.layer < 0 || sp.layer >= num_layers || (i > 0 && sp.layer <= steps_h[i - 1].layer)) return APACK_EINVAL;
    if (!sp.q || !sp.k_out || !sp.v_out || !sp.keep_idx || !sp.modality_out || !sp.new_cu_seqlens_h)
      return APACK_EINVAL;
    if (hidden && !sp.hidden_out) return APACK_EINVAL;
    // the step's queries are read by TMA: 16-byte aligned device memory
    if ((reinterpret_cast<uintptr_t>(sp.q) & 15) || in_host_memory(sp.q)) return APACK_EINVAL;
    if (i == 0) {
      p.cu.assign(seqs->cu_seqlens_h, seqs->cu_seqlens_h + B + 1);
      p.na.assign(seqs->n_audio_h, seqs->n_audio_h + B);
      p.nv.assign(seqs->n_visual_h, seqs->n_visual_h + B);
      p.seqs = *seqs;
      p.k = k_cache;
      p.v = v_cache;
      p.hidden = hidden;
      p.kv_layer_stride = kv_layer_stride;
    } else {
      const StepPlan &q = plan[i - 1];
      const apack_step &prev = steps_h[i - 1];
      p.cu.assign(prev.new_cu_seqlens_h, prev.new_cu_seqlens_h + B + 1);
      p.na.resize(B);
      p.nv.resize(B);
      for (int b = 0; b < B; ++b) {
        p.na[b] = q.counts[2 * b];
        p.nv[b] = q.counts[2 * b + 1];
      }
      p.seqs = *seqs;
      p.seqs.modality = prev.modality_out;
      const int64_t skip = sp.layer - prev.layer;
      p.k = static_cast<const uint8_t *>(prev.k_out) + skip * prev.kv_out_layer_stride;
      p.v = static_cast<const uint8_t *>(prev.v_out) + skip * prev.kv_out_layer_stride;
      p.hidden = prev.hidden_out;
      p.kv_layer_stride = prev.kv_out_layer_stride;
    }
    p.seqs.cu_seqlens_h = p.cu.data();
    p.seqs.n_audio_h = p.na.data();
    p.seqs.n_visual_h = p.nv.data();
    int64_t Ti = 0, NQi = 0;
    st = validate_seqs(&p.seqs, &Ti, &NQi);
    if (st != APACK_OK) return st;
    if (!ws_ok(&p.seqs, ws, ws_bytes)) return ws ? APACK_EWORKSPACE : APACK_EINVAL;
    p.counts.assign(2 * static_cast<size_t>(B), 0);
    st = counts_and_offsets(&p.seqs, sp.keep_ratio_h, sp.keep_count_h, select_mode, p.counts.data(),
                            sp.new_cu_seqlens_h);
    if (st != APACK_OK) return st;
    const int64_t n_out = sp.new_cu_seqlens_h[B];
    const int32_t n_layers = num_layers - sp.layer;
    if (n_layers > 1 && (p.kv_layer_stride < Ti * row || sp.kv_out_layer_stride < n_out * row)) return APACK_EINVAL;
    // in place: both caches together, with the input's slab stride
    if ((sp.k_out == p.k) != (sp.v_out == p.v) || (sp.k_out == p.k && sp.kv_out_layer_stride != p.kv_layer_stride))
      return APACK_EINVAL;
    // compaction: K/V of layers [l_i, L), hidden, extra planes, in one launch
    if (sp.num_extra < 0 || (sp.num_extra > 0 && !sp.extra_planes_h)) return APACK_EINVAL;
    p.planes.reserve(3 + static_cast<size_t>(sp.num_extra));
    p.planes.push_back(plane(p.k, sp.k_out, p.kv_layer_stride, sp.kv_out_layer_stride, row, n_layers));
    p.planes.push_back(plane(p.v, sp.v_out, p.kv_layer_stride, sp.kv_out_layer_stride, row, n_layers));
    if (p.hidden) p.planes.push_back(plane(p.hidden, sp.hidden_out, 0, 0, hidden_dim * 2, 1));
    for (int e = 0; e < sp.num_extra; ++e) p.planes.push_back(sp.extra_planes_h[e]);
    st = run_compact(sp.keep_idx, n_out, p.planes.data(), static_cast<int32_t>(p.planes.size()), err, nullptr, true);
    if (st != APACK_OK) return st;
  }

  cudaStream_t M = static_cast<cudaStream_t>(stream);
  auto mark = [&](int step, int k) {
    if (stage_events_h && stage_events_h[4 * step + k])
      cudaEventRecord(static_cast<cudaEvent_t>(stage_events_h[4 * step + k]), M);
  };
  for (int i = 0; i < num_steps; ++i) {
    const apack_step &sp = steps_h[i];
    const StepPlan &p = plan[i];
    mark(i, 0);
    st = run_score(&p.seqs, sp.q, p.k, row, scores, ws, M);
    if (st != APACK_OK) return st;
    mark(i, 1);
    st = run_select(&p.seqs, scores, p.counts.data(), select_mode, sp.keep_idx, sp.modality_out, nullptr,
                    sp.new_cu_seqlens, ws, M);
    if (st != APACK_OK) return st;
    mark(i, 2);
    st = run_compact(sp.keep_idx, sp.new_cu_seqlens_h[B], p.planes.data(), static_cast<int32_t>(p.planes.size()),
                     err, M);
    if (st != APACK_OK) return st;
    mark(i, 3);
  }
  return APACK_OK;
}

struct apack_graph_s {
  cudaGraphExec_t exec;
  uint64_t launches;     // kernels per replay
};

apack_status apack_prune_schedule_graph(const apack_seqs *seqs, int32_t num_layers, const void *k_cache,
                                        const void *v_cache, int64_t kv_layer_stride, const void *hidden,
                                        int64_t hidden_dim, int32_t select_mode, const apack_step *steps_h,
                                        int32_t num_steps, float *scores, void *ws, size_t ws_bytes,
                                        apack_graph *graph_out) {
  if (!graph_out) return APACK_EINVAL;
  *graph_out = nullptr;
  cudaStream_t cs = nullptr;
  if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) return APACK_ECUDA;
  const uint64_t before = apack_launch_count();
  if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
    cudaStreamDestroy(cs);
    return APACK_ECUDA;
  }
  apack_status st = apack_prune_schedule(seqs, num_layers, k_cache, v_cache, kv_layer_stride, hidden, hidden_dim,
                                         select_mode, steps_h, num_steps, scores, ws, ws_bytes, nullptr, cs);
  cudaGraph_t g = nullptr;
  const cudaError_t ce = cudaStreamEndCapture(cs, &g);
  const uint64_t captured = apack_launch_count() - before;
  count_launches(0 - captured);                 // nothing ran: captured launches count when replayed
  cudaStreamDestroy(cs);
  if (st == APACK_OK && (ce != cudaSuccess || !g)) st = APACK_ECUDA;
  cudaGraphExec_t exec = nullptr;
  if (st == APACK_OK && cudaGraphInstantiate(&exec, g, 0) != cudaSuccess) st = APACK_ECUDA;
  if (g) cudaGraphDestroy(g);
  cudaGetLastError();                           // a refused capture leaves no sticky error behind
  if (st != APACK_OK) {
    if (exec) cudaGraphExecDestroy(exec);
    return st;
  }
  apack_graph h = new (std::nothrow) apack_graph_s{exec, captured};
  if (!h) {
    cudaGraphExecDestroy(exec);
    return APACK_ECUDA;
  }
  *graph_out = h;
  return APACK_OK;
}

apack_status apack_graph_launch(apack_graph graph, void *stream) {
  if (!graph) return APACK_EINVAL;
  if (cudaGraphLaunch(graph->exec, static_cast<cudaStream_t>(stream)) != cudaSuccess) return APACK_ECUDA;
  count_launches(graph->launches);
  return APACK_OK;
}

apack_status apack_graph_destroy(apack_graph graph) {
  if (!graph) return APACK_OK;
  const cudaError_t e = cudaGraphExecDestroy(graph->exec);
  delete graph;
  return e == cudaSuccess ? APACK_OK : APACK_ECUDA;
}

}  // extern "C"
