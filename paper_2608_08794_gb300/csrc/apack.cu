// apack.cu -- the C ABI of include/apack.h: argument checks, workspace planning and the
// sequencing of one pruning step (Sec. 3.2; Algorithm 1, one iteration of the inner-LLM loop).
#include <atomic>
#include <cmath>
#include <cstring>
#include <vector>

#include "internal.cuh"

namespace apack {

namespace {
std::atomic<uint64_t> g_launches{0};
std::atomic<int> g_sm_count[64];   // per device; 0 = not read yet
}  // namespace

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

apack_status check_cuda(cudaError_t e) { return e == cudaSuccess ? APACK_OK : APACK_ECUDA; }

bool in_host_memory(const void *p) {
  if (!p) return false;
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeHost;
}

int device_sm_count() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 148;
  if (dev < 64) {
    const int cached = g_sm_count[dev].load(std::memory_order_relaxed);
    if (cached > 0) return cached;
  }
  int n = 0;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 148;
  if (dev < 64) g_sm_count[dev].store(n, std::memory_order_relaxed);
  return n;
}

apack_status validate_seqs(const apack_seqs *s, int64_t *total_tokens, int64_t *total_qrows) {
  if (!s || s->num_seqs < 1 || s->num_seqs > APACK_MAX_SEQS) return APACK_EINVAL;
  if (!s->cu_seqlens_h || !s->cu_qlens_h || !s->n_audio_h || !s->n_visual_h) return APACK_EINVAL;
  if (s->head_dim != APACK_HEAD_DIM) return APACK_EUNSUPPORTED;
  if (s->num_q_heads < 1 || s->num_kv_heads < 1 || s->num_q_heads % s->num_kv_heads != 0) return APACK_EINVAL;
  if (s->cu_seqlens_h[0] != 0 || s->cu_qlens_h[0] != 0) return APACK_EINVAL;
  if (s->softmax_domain != APACK_SOFTMAX_MM && s->softmax_domain != APACK_SOFTMAX_CAUSAL_ROW) return APACK_EINVAL;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int64_t len = static_cast<int64_t>(s->cu_seqlens_h[b + 1]) - s->cu_seqlens_h[b];
    const int64_t nq = static_cast<int64_t>(s->cu_qlens_h[b + 1]) - s->cu_qlens_h[b];
    if (len < 0 || nq < 0) return APACK_EINVAL;
    if (s->softmax_domain == APACK_SOFTMAX_CAUSAL_ROW && nq > len) return APACK_EINVAL;   // rows are tokens
    if (s->softmax_domain == APACK_SOFTMAX_CAUSAL_ROW && s->q_start_h &&
        (s->q_start_h[b] < 0 || static_cast<int64_t>(s->q_start_h[b]) + nq > len))
      return APACK_EINVAL;
    if (s->n_audio_h[b] < 0 || s->n_visual_h[b] < 0 ||
        static_cast<int64_t>(s->n_audio_h[b]) + s->n_visual_h[b] > len)
      return APACK_EINVAL;
  }
  const int64_t T = s->cu_seqlens_h[s->num_seqs];
  if (T > 0 && !s->modality) return APACK_EINVAL;
  *total_tokens = T;
  *total_qrows = s->cu_qlens_h[s->num_seqs];
  return APACK_OK;
}

int32_t query_position(const apack_seqs *s, int b) {
  const int32_t len = s->cu_seqlens_h[b + 1] - s->cu_seqlens_h[b];
  const int32_t nq = s->cu_qlens_h[b + 1] - s->cu_qlens_h[b];
  return s->q_start_h ? s->q_start_h[b] : len - nq;
}

WsLayout workspace_layout(const apack_seqs *s) {
  WsLayout L{};
  const int64_t NQ = s->cu_qlens_h[s->num_seqs];
  const int64_t T = s->cu_seqlens_h[s->num_seqs];
  const int G = s->num_q_heads / s->num_kv_heads;
  int64_t chunks = 0, qp_rows = 0;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int64_t rows = static_cast<int64_t>(G) * (s->cu_qlens_h[b + 1] - s->cu_qlens_h[b]);
    chunks += static_cast<int64_t>(s->num_kv_heads) * ((rows + 127) / 128);
    qp_rows += static_cast<int64_t>(s->num_kv_heads) * ((rows + 255) / 256) * 256;
  }
  auto up = [](size_t x) { return (x + 1023) & ~static_cast<size_t>(1023); };
  L.err_off = 0;
  if (narrow_score_applies(s)) {
    size_t lf = 0, pf = 0, ef = 0;
    narrow_layout(s, &lf, &pf, &ef);
    L.narrow = true;
    L.nlog_off = 1024;
    L.npart_off = up(L.nlog_off + lf * sizeof(float));
    L.nlse_off = up(L.npart_off + pf * sizeof(float2));
    L.total = up(L.nlse_off + ef * sizeof(float));
    return L;
  }
  L.part_off = 1024;
  const size_t part_bytes = static_cast<size_t>(kMaxSplits) * NQ * s->num_q_heads * sizeof(float2);
  L.lse_off = up(L.part_off + part_bytes);
  L.lse_chunks = chunks;
  L.qp_off = up(L.lse_off + static_cast<size_t>(qp_rows) * sizeof(float));
  L.qp_rows = qp_rows;
  L.gsum_off = up(L.qp_off + static_cast<size_t>(qp_rows) * 256);
  int64_t key_blocks = 0;   // 256-key blocks of the sequences that have query rows
  for (int b = 0; b < s->num_seqs; ++b)
    if (s->cu_qlens_h[b + 1] > s->cu_qlens_h[b])
      key_blocks += (static_cast<int64_t>(s->cu_seqlens_h[b + 1]) - s->cu_seqlens_h[b] + 255) / 256;
  L.mask_off = up(L.gsum_off + static_cast<size_t>(s->num_kv_heads) * T * sizeof(float));
  L.total = up(L.mask_off + static_cast<size_t>(key_blocks) * 32);
  return L;
}

}  // namespace apack

using namespace apack;

namespace {

int32_t keep_count_rule(float ratio, int32_t n) {
  // k = min(n, ceil(round(r * 1e6) * n / 1e6)) in integer arithmetic.
  const int64_t num = static_cast<int64_t>(std::floor(static_cast<double>(ratio) * 1e6 + 0.5));
  const int64_t k = (num * n + 999999) / 1000000;
  return static_cast<int32_t>(k < n ? k : n);
}

bool ratios_ok(const apack_seqs *s, const float *r, int32_t mode) {
  for (int b = 0; b < s->num_seqs; ++b)
    for (int m = 0; m < (mode == APACK_SELECT_JOINT ? 1 : 2); ++m) {
      const float x = r[2 * b + m];
      if (!(x >= 0.f && x <= 1.f)) return false;
    }
  return true;
}

}  // namespace

namespace apack {

apack_status counts_and_offsets(const apack_seqs *s, const float *ratio_h, const int32_t *count_h, int32_t mode,
                                 int32_t *k_out, int32_t *cu_out) {
  if (mode != APACK_SELECT_PER_MODALITY && mode != APACK_SELECT_JOINT) return APACK_EINVAL;
  if (!count_h) {
    if (!ratio_h || !ratios_ok(s, ratio_h, mode)) return APACK_EINVAL;
  }
  int64_t acc = 0;
  if (cu_out) cu_out[0] = 0;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int32_t na = s->n_audio_h[b], nv = s->n_visual_h[b];
    const int32_t len = s->cu_seqlens_h[b + 1] - s->cu_seqlens_h[b];
    int32_t k0, k1;
    if (count_h) {
      k0 = count_h[2 * b];
      k1 = mode == APACK_SELECT_JOINT ? 0 : count_h[2 * b + 1];
    } else if (mode == APACK_SELECT_JOINT) {
      k0 = keep_count_rule(ratio_h[2 * b], na + nv);
      k1 = 0;
    } else {
      k0 = keep_count_rule(ratio_h[2 * b], na);
      k1 = keep_count_rule(ratio_h[2 * b + 1], nv);
    }
    if (mode == APACK_SELECT_JOINT) {
      if (k0 < 0 || k0 > na + nv) return APACK_EINVAL;
    } else if (k0 < 0 || k0 > na || k1 < 0 || k1 > nv) {
      return APACK_EINVAL;
    }
    if (k_out) {
      k_out[2 * b] = k0;
      k_out[2 * b + 1] = k1;
    }
    acc += len - na - nv + k0 + k1;
    if (cu_out) cu_out[b + 1] = static_cast<int32_t>(acc);
  }
  return APACK_OK;
}

bool ws_ok(const apack_seqs *s, const void *ws, size_t bytes) {
  if (!ws || (reinterpret_cast<uintptr_t>(ws) & 255)) return false;
  return bytes >= workspace_layout(s).total;
}

}  // namespace apack

extern "C" {

apack_status apack_workspace_size(const apack_seqs *seqs, size_t *bytes) {
  int64_t T = 0, NQ = 0;
  if (!bytes) return APACK_EINVAL;
  const apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  *bytes = workspace_layout(seqs).total;
  return APACK_OK;
}

apack_status apack_keep_counts(const apack_seqs *seqs, const float *keep_ratio_h, int32_t select_mode,
                               int32_t *keep_count_h, int32_t *new_cu_seqlens_h) {
  int64_t T = 0, NQ = 0;
  const apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (!keep_ratio_h) return APACK_EINVAL;
  return counts_and_offsets(seqs, keep_ratio_h, nullptr, select_mode, keep_count_h, new_cu_seqlens_h);
}

apack_status apack_score(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                         float *scores, void *ws, size_t ws_bytes, void *stream) {
  int64_t T = 0, NQ = 0;
  const apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (!ws_ok(seqs, ws, ws_bytes)) return ws ? APACK_EWORKSPACE : APACK_EINVAL;
  if (in_host_memory(k) || in_host_memory(q)) return APACK_EINVAL;   // read by TMA: device memory only
  return run_score(seqs, q, k, k_token_stride, scores, ws, static_cast<cudaStream_t>(stream));
}

apack_status apack_select(const apack_seqs *seqs, const float *scores, const float *keep_ratio_h,
                          const int32_t *keep_count_h, int32_t select_mode, int32_t *keep_idx,
                          uint8_t *modality_out, int32_t *dst_of_src, int32_t *new_cu_seqlens, void *ws,
                          size_t ws_bytes, void *stream) {
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (!ws_ok(seqs, ws, ws_bytes)) return ws ? APACK_EWORKSPACE : APACK_EINVAL;
  // counts from the ratios when none are given (the rule of apack_keep_counts), checked either way
  std::vector<int32_t> counts(2 * static_cast<size_t>(seqs->num_seqs));
  st = counts_and_offsets(seqs, keep_ratio_h, keep_count_h, select_mode, counts.data(), nullptr);
  if (st != APACK_OK) return st;
  return run_select(seqs, scores, counts.data(), select_mode, keep_idx, modality_out, dst_of_src, new_cu_seqlens, ws,
                    static_cast<cudaStream_t>(stream));
}

apack_status apack_compact(const int32_t *keep_idx, int64_t n_out, const apack_plane *planes_h, int32_t num_groups,
                           void *ws, void *stream) {
  if (ws && (reinterpret_cast<uintptr_t>(ws) & 255)) return APACK_EINVAL;
  return run_compact(keep_idx, n_out, planes_h, num_groups, static_cast<DeviceError *>(ws),
                     static_cast<cudaStream_t>(stream));
}

apack_status apack_prune_step(const apack_seqs *seqs, int32_t layer, int32_t num_layers, const void *q,
                              const void *k_cache, const void *v_cache, int64_t kv_layer_stride, const void *hidden,
                              int64_t hidden_dim, const float *keep_ratio_h, const int32_t *keep_count_h,
                              int32_t select_mode, void *k_out, void *v_out, int64_t kv_out_layer_stride,
                              void *hidden_out, const apack_plane *extra_planes_h, int32_t num_extra,
                              uint8_t *modality_out, int32_t *keep_idx, int32_t *new_cu_seqlens_h,
                              int32_t *new_cu_seqlens, float *scores, void *ws, size_t ws_bytes,
                              void *const *stage_events_h, void *stream) {
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (layer < 0 || num_layers <= layer || !k_cache || !v_cache || !k_out || !v_out || !keep_idx || !scores ||
      !new_cu_seqlens_h || num_extra < 0 || (num_extra > 0 && !extra_planes_h))
    return APACK_EINVAL;
  if (hidden && (!hidden_out || hidden_dim <= 0)) return APACK_EINVAL;
  if (!ws_ok(seqs, ws, ws_bytes)) return ws ? APACK_EWORKSPACE : APACK_EINVAL;
  if (in_host_memory(k_cache) || in_host_memory(q)) return APACK_EINVAL;   // scored by TMA: device memory
  // in place: both caches together, with the input's slab stride (checked before any launch)
  if ((k_out == k_cache) != (v_out == v_cache) || (k_out == k_cache && kv_out_layer_stride != kv_layer_stride))
    return APACK_EINVAL;
  const int64_t row = static_cast<int64_t>(seqs->num_kv_heads) * APACK_HEAD_DIM * 2;
  const int32_t n_layers = num_layers - layer;
  if (n_layers > 1 && (kv_layer_stride < T * row || kv_out_layer_stride < row)) return APACK_EINVAL;
  std::vector<int32_t> counts(2 * static_cast<size_t>(seqs->num_seqs));
  st = counts_and_offsets(seqs, keep_ratio_h, keep_count_h, select_mode, counts.data(), new_cu_seqlens_h);
  if (st != APACK_OK) return st;
  const int64_t n_out = new_cu_seqlens_h[seqs->num_seqs];
  if (n_layers > 1 && kv_out_layer_stride < n_out * row) return APACK_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // compaction groups: K/V of layers [layer, num_layers), hidden, extra planes
  std::vector<apack_plane> planes;
  planes.reserve(3 + static_cast<size_t>(num_extra));
  apack_plane kp{};
  kp.src = k_cache;
  kp.dst = k_out;
  kp.src_plane_stride = kv_layer_stride;
  kp.dst_plane_stride = kv_out_layer_stride;
  kp.src_row_stride = row;
  kp.dst_row_stride = row;
  kp.row_bytes = row;
  kp.num_planes = n_layers;
  planes.push_back(kp);
  apack_plane vp = kp;
  vp.src = v_cache;
  vp.dst = v_out;
  planes.push_back(vp);
  if (hidden) {
    apack_plane hp{};
    hp.src = hidden;
    hp.dst = hidden_out;
    hp.src_row_stride = hp.dst_row_stride = hp.row_bytes = hidden_dim * 2;
    hp.num_planes = 1;
    planes.push_back(hp);
  }
  for (int i = 0; i < num_extra; ++i) planes.push_back(extra_planes_h[i]);
  DeviceError *err = reinterpret_cast<DeviceError *>(static_cast<uint8_t *>(ws) + workspace_layout(seqs).err_off);
  // every argument of the compaction is checked before the first launch of the step
  st = run_compact(keep_idx, n_out, planes.data(), static_cast<int32_t>(planes.size()), err, s, true);
  if (st != APACK_OK) return st;
  auto mark = [&](int i) {
    if (stage_events_h && stage_events_h[i]) cudaEventRecord(static_cast<cudaEvent_t>(stage_events_h[i]), s);
  };
  mark(0);
  st = run_score(seqs, q, k_cache, row, scores, ws, s);
  if (st != APACK_OK) return st;
  mark(1);
  st = run_select(seqs, scores, counts.data(), select_mode, keep_idx, modality_out, nullptr, new_cu_seqlens, ws, s);
  if (st != APACK_OK) return st;
  mark(2);
  st = run_compact(keep_idx, n_out, planes.data(), static_cast<int32_t>(planes.size()), err, s);
  if (st != APACK_OK) return st;
  mark(3);
  return APACK_OK;
}

apack_status apack_device_error(const void *ws, void *stream, int32_t *code_out, int32_t clear) {
  if (!ws || !code_out) return APACK_EINVAL;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  DeviceError e{};
  if (cudaStreamSynchronize(s) != cudaSuccess) return APACK_ECUDA;
  if (cudaMemcpy(&e, ws, sizeof(e), cudaMemcpyDeviceToHost) != cudaSuccess) return APACK_ECUDA;
  *code_out = e.code;
  if (clear && e.code != 0) {
    DeviceError z{};
    if (cudaMemcpy(const_cast<void *>(ws), &z, sizeof(z), cudaMemcpyHostToDevice) != cudaSuccess)
      return APACK_ECUDA;
  }
  return APACK_OK;
}

uint64_t apack_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char *apack_status_string(apack_status status) {
  switch (status) {
    case APACK_OK: return "ok";
    case APACK_EINVAL: return "invalid argument";
    case APACK_ECUDA: return "CUDA error";
    case APACK_EWORKSPACE: return "workspace too small";
    case APACK_ETIMEOUT: return "device wait timed out";
    case APACK_EDEVICE: return "device data disagree with host counts";
    case APACK_EUNSUPPORTED: return "unsupported shape or mode";
    default: return "unknown status";
  }
}

}  // extern "C"
