// decode.cu -- attention of one decode token over a (compacted) KV cache: the cost the
// inner-LLM pruning shortens for every autoregressive step (Sec. 3.2, last sentence;
// App. G, decoding throughput).
//
//   out[b, h] = sum_j softmax_j(q[b, h] . k[j, g(h)] / sqrt(128)) v[j, g(h)],
//   g(h) = h / (Hq / Hkv), j over every cached token of sequence b.
//
// Split-KV in two launches.  With Hkv 2 or 4 and at most 8 query rows per KV head the chunk
// kernel is the tensor-core one of decode_tc.cu (its CTAs claim the sequence's stages from a
// counter, so the keys' grouping into partials varies from call to call); otherwise:
//   chunk kernel:   one CTA per (sequence, chunk of about T / #SMs keys).  K and V rows
//                   stream into a 3-stage shared-memory ring by bulk async copies (issued
//                   by one lane).  Each of 16 warps works on KV head
//                   w % Hkv and one group of 8 keys of every stage; lane l owns features
//                   [4l, 4l + 4) of that head for all G <= 8 query rows of the head group.
//                   Per 8 keys: logits by a reduce-scatter of the 8 row partials over the
//                   warp (the lane's query rows are stored in an order that makes every
//                   step a plain shuffle and add), online max and sum per row,
//                   probabilities handed to all lanes through shared memory, P.V
//                   accumulated in registers.  The warps of a head merge in shared memory;
//                   the CTA writes (max, sum, o[128]) per query head.
//   combine kernel: one CTA per (sequence, query head) merges the chunks in order.
// K and V are read once: the chunk kernel is HBM-bound.  The CUDA-core path's merges run in a
// fixed order, so its output is deterministic; the combine merges any path's partials in a
// fixed order.
#include <algorithm>
#include <cmath>

#include "decode_plan.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kDecConsumers = 16;                 // warps per CTA; lane 0 of the last also loads
constexpr int kDecThreads = kDecConsumers * 32;
constexpr int kDecStages = 3;                     // shared-memory ring of K/V stages
constexpr int kStageBytes = 32768;                // K (and V) bytes per stage: 128 / Hkv tokens
constexpr int kDecRows = 8;                       // query rows per KV head group (G <= 8)
constexpr size_t kDecSmem = static_cast<size_t>(kDecStages) * 2 * kStageBytes + 2 * kDecStages * sizeof(uint64_t) +
                            (kDecConsumers * 8 * kDecRows + kDecConsumers * kDecRows) * sizeof(float) + 16;
constexpr int kDecCombineThreads = 512;
constexpr int kDecCombineWarps = kDecCombineThreads / 32;

__device__ __forceinline__ void bf16x4_to_f32(const uint2 &w, float (&f)[4]) {
  f[0] = __uint_as_float(w.x << 16);
  f[1] = __uint_as_float(w.x & 0xFFFF0000u);
  f[2] = __uint_as_float(w.y << 16);
  f[3] = __uint_as_float(w.y & 0xFFFF0000u);
}

// Merge (m2, l2, o2) into (m1, l1, o1) (log2 units).
__device__ __forceinline__ void merge_state(float &m1, float &l1, float (&o1)[4], float m2, float l2,
                                            const float (&o2)[4]) {
  if (m2 == -INFINITY) return;
  const float mn = fmaxf(m1, m2);
  const float a = ex2_approx(m1 - mn), b = ex2_approx(m2 - mn);   // m1 = -inf gives a = 0
  l1 = l1 * a + l2 * b;
#pragma unroll
  for (int e = 0; e < 4; ++e) o1[e] = o1[e] * a + o2[e] * b;
  m1 = mn;
}

// q: bf16 [nseq][Hq][128] of this launch's sequences.  Partials per (chunk, query head):
// opart [chunks][Hq][128], mlpart [chunks][Hq] = (max, sum) in log2 units.
//
// K and V rows stream into a ring of kDecStages shared-memory stages by bulk async copies;
// a stage holds kStageBytes of K and of V (128 / Hkv tokens).  Warp w takes KV head w % Hkv
// and the group of 8 keys (w / Hkv) of every stage, so all 16 warps consume a stage
// together.  Lane 0 of the last warp is also the loader: it issues the first stages, and
// after its own group of stage n, once every warp has released stage n, it refills that
// stage's slot with stage n + kDecStages.
__device__ __forceinline__ void decode_issue_stage(const DecSeq &sq, const uint8_t *k, const uint8_t *v,
                                                   int64_t kv_stride, int64_t row, int stage_tok, int tb, int te,
                                                   int n, uint8_t *stage_base, uint64_t *full) {
  const int slot = n % kDecStages;
  const int t = tb + n * stage_tok;
  const int cnt = min(stage_tok, te - t);
  uint8_t *ks = stage_base + static_cast<size_t>(slot) * 2 * kStageBytes;
  uint8_t *vs = ks + kStageBytes;
  mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(2 * cnt * row));
  const int64_t g0 = static_cast<int64_t>(sq.t0) + t;
  if (kv_stride == row) {   // dense rows: one copy per tensor
    bulk_load(ks, k + g0 * kv_stride, static_cast<uint32_t>(cnt * row), &full[slot]);
    bulk_load(vs, v + g0 * kv_stride, static_cast<uint32_t>(cnt * row), &full[slot]);
  } else {
    for (int r = 0; r < cnt; ++r) {
      bulk_load(ks + r * row, k + (g0 + r) * kv_stride, static_cast<uint32_t>(row), &full[slot]);
      bulk_load(vs + r * row, v + (g0 + r) * kv_stride, static_cast<uint32_t>(row), &full[slot]);
    }
  }
}

__global__ void __launch_bounds__(kDecThreads, 1)
    decode_chunk_kernel(const __grid_constant__ DecPlan plan, const uint16_t *__restrict__ q,
                        const uint8_t *__restrict__ k, const uint8_t *__restrict__ v, int64_t kv_stride,
                        float *__restrict__ opart, float2 *__restrict__ mlpart, DeviceError *err) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");   // the combine may be scheduled
  extern __shared__ __align__(1024) uint8_t dsmem[];
  uint8_t *stage_base = dsmem;                                               // [kDecStages][K | V]
  uint64_t *full = reinterpret_cast<uint64_t *>(dsmem + kDecStages * 2 * kStageBytes);
  uint64_t *empty = full + kDecStages;
  float *ps = reinterpret_cast<float *>(empty + kDecStages);                 // [warp][key][row]
  float *sc = ps + kDecConsumers * 8 * kDecRows;                             // [warp][row]
  int *abort_flag = reinterpret_cast<int *>(sc + kDecConsumers * kDecRows);
  const int c = blockIdx.x;
  const int s = find_chunk_seq(plan, c);
  const DecSeq &sq = plan.seq[s];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int G = plan.group, hkv = plan.hkv;
  const int64_t row = static_cast<int64_t>(hkv) * 256;
  const int stage_tok = kStageBytes / static_cast<int>(row);
  const int tb = (c - sq.chunk_begin) * plan.chunk;
  const int te = min(sq.len, tb + plan.chunk);
  const int nst = (te - tb + stage_tok - 1) / stage_tok;
  const bool loader = warp == kDecConsumers - 1 && lane == 0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kDecStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kDecConsumers);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int *abort_v = abort_flag;
  int issued = 0;
  if (loader)
    for (; issued < kDecStages && issued < nst; ++issued)
      decode_issue_stage(sq, k, v, kv_stride, row, stage_tok, tb, te, issued, stage_base, full);

  const int h = warp % hkv, grp = warp / hkv;
  const int cl = (lane >> 2) & 7;       // after the reduce-scatter this lane holds row cl
  float qf[kDecRows][4];                // query rows, lane-permuted: slot j holds row j ^ cl
  const uint16_t *qg = q + (static_cast<int64_t>(s) * plan.hq + h * G) * 128 + lane * 4;
#pragma unroll
  for (int j = 0; j < kDecRows; ++j) {
    const int r = j ^ cl;
    uint2 w = make_uint2(0, 0);
    if (r < G) w = __ldg(reinterpret_cast<const uint2 *>(qg + r * 128));
    bf16x4_to_f32(w, qf[j]);
  }
  float o[kDecRows][4];
#pragma unroll
  for (int j = 0; j < kDecRows; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_own = -INFINITY, l_own = 0.f;
  float *wps = ps + warp * 8 * kDecRows;
  float *wsc = sc + warp * kDecRows;
  for (int n = 0; n < nst; ++n) {
    const int slot = n % kDecStages;
    // the decision to go on is warp-uniform: every lane waited, and all must have succeeded
    if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], (n / kDecStages) & 1u, kWaitLimitNs))) {
      if (lane == 0) {
        raise_device_error(err, APACK_ETIMEOUT, 62, c, n);
        *abort_v = 1;
      }
      break;
    }
    const int t = tb + n * stage_tok + grp * 8;
    const int valid = min(8, te - t);
    if (valid > 0) {
      const uint8_t *ks = stage_base + static_cast<size_t>(slot) * 2 * kStageBytes +
                          static_cast<size_t>(grp) * 8 * row + h * 256 + lane * 8;
      const uint8_t *vs = ks + kStageBytes;
      float x[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float kf[4];
        bf16x4_to_f32(i < valid ? *reinterpret_cast<const uint2 *>(ks + i * row) : make_uint2(0, 0), kf);
        float acc[kDecRows];
#pragma unroll
        for (int j = 0; j < kDecRows; j += 2) {
          float2 a = make_float2(0.f, 0.f);
#pragma unroll
          for (int e = 0; e < 4; ++e) a = ffma2(make_float2(kf[e], kf[e]), make_float2(qf[j][e], qf[j + 1][e]), a);
          acc[j] = a.x;
          acc[j + 1] = a.y;
        }
        // slot e and the partner's slot e + half hold the same row at every level
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e + 4], 16);
#pragma unroll
        for (int e = 0; e < 2; ++e) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e + 2], 8);
        acc[0] += __shfl_xor_sync(0xffffffffu, acc[1], 4);
        acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], 2);
        acc[0] += __shfl_xor_sync(0xffffffffu, acc[0], 1);
        x[i] = i < valid ? acc[0] * plan.scale2 : -INFINITY;
      }
      // online softmax of row cl over these keys (key 0 of the group is valid)
      float cm = x[0];
#pragma unroll
      for (int i = 1; i < 8; ++i) cm = fmaxf(cm, x[i]);
      const float mn = fmaxf(m_own, cm);
      const float scale = ex2_approx(m_own - mn);
      float psum = 0.f;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float p = ex2_approx(x[i] - mn);
        psum += p;
        wps[i * kDecRows + cl] = p;        // the four lanes of a row write the same value
      }
      wsc[cl] = scale;
      l_own = l_own * scale + psum;
      m_own = mn;
      __syncwarp();
      {
        const float4 sa = *reinterpret_cast<const float4 *>(wsc);
        const float4 sb = *reinterpret_cast<const float4 *>(wsc + 4);
        const float sr[8] = {sa.x, sa.y, sa.z, sa.w, sb.x, sb.y, sb.z, sb.w};
#pragma unroll
        for (int j = 0; j < kDecRows; ++j)
#pragma unroll
          for (int e = 0; e < 4; ++e) o[j][e] *= sr[j];
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float vf[4];
        bf16x4_to_f32(i < valid ? *reinterpret_cast<const uint2 *>(vs + i * row) : make_uint2(0, 0), vf);
        const float4 pa = *reinterpret_cast<const float4 *>(wps + i * kDecRows);
        const float4 pb = *reinterpret_cast<const float4 *>(wps + i * kDecRows + 4);
        const float pr[8] = {pa.x, pa.y, pa.z, pa.w, pb.x, pb.y, pb.z, pb.w};
#pragma unroll
        for (int j = 0; j < kDecRows; j += 2)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float2 r2 = ffma2(make_float2(pr[j], pr[j + 1]), make_float2(vf[e], vf[e]),
                                    make_float2(o[j][e], o[j + 1][e]));
            o[j][e] = r2.x;
            o[j + 1][e] = r2.y;
          }
      }
    }
    __syncwarp();                        // this warp is done with the stage and its scratch
    if (lane == 0) mbar_arrive(&empty[slot]);
    if (loader && issued < nst) {
      // every warp has released stage n: refill its slot
      if (!mbar_wait(&empty[slot], (n / kDecStages) & 1u, kWaitLimitNs)) {
        raise_device_error(err, APACK_ETIMEOUT, 61, c, n);
        *abort_v = 1;
      } else {
        decode_issue_stage(sq, k, v, kv_stride, row, stage_tok, tb, te, issued, stage_base, full);
        ++issued;
      }
    }
    __syncwarp();
    if (*abort_v) break;
  }
  // after an abort, stages may still be in flight: wait for them (bounded) before the
  // shared memory is reused or the CTA exits
  if (loader && *abort_v)
    for (int n = max(0, issued - kDecStages); n < issued; ++n)
      mbar_wait(&full[n % kDecStages], (n / kDecStages) & 1u, kWaitLimitNs / 4);
  __syncthreads();
  if (*abort_v) return;
  // merge the warps of each head in group order; the stages are free now
  float *wo = reinterpret_cast<float *>(stage_base);                   // [warp][row][128]
  float2 *wml = reinterpret_cast<float2 *>(wo + kDecConsumers * kDecRows * 128);
#pragma unroll
  for (int j = 0; j < kDecRows; ++j)
    *reinterpret_cast<float4 *>(wo + (warp * kDecRows + j) * 128 + lane * 4) =
        make_float4(o[j][0], o[j][1], o[j][2], o[j][3]);
  if ((lane & 3) == 0) wml[warp * kDecRows + cl] = make_float2(m_own, l_own);
  __syncthreads();
  if (grp == 0) {
    for (int j = 0; j < G; ++j) {
      float m1 = wml[warp * kDecRows + j].x, l1 = wml[warp * kDecRows + j].y;
      const float4 a = *reinterpret_cast<const float4 *>(wo + (warp * kDecRows + j) * 128 + lane * 4);
      float o1[4] = {a.x, a.y, a.z, a.w};
      for (int g2 = 1; g2 < kDecConsumers / hkv; ++g2) {
        const int w2 = g2 * hkv + h;
        const float2 ml2 = wml[w2 * kDecRows + j];
        const float4 b = *reinterpret_cast<const float4 *>(wo + (w2 * kDecRows + j) * 128 + lane * 4);
        const float o2[4] = {b.x, b.y, b.z, b.w};
        merge_state(m1, l1, o1, ml2.x, ml2.y, o2);
      }
      const int64_t hq_idx = static_cast<int64_t>(c) * plan.hq + h * G + j;
      *reinterpret_cast<float4 *>(opart + hq_idx * 128 + lane * 4) = make_float4(o1[0], o1[1], o1[2], o1[3]);
      if (lane == 0) mlpart[hq_idx] = make_float2(m1, l1);
    }
  }
}

// One CTA per (sequence, query head): merge the sequence's chunks.  Warp w folds chunks
// w, w + 16, w + 32, ... in that order (lane: features [4 lane, 4 lane + 4)); the warps
// then merge in warp order.  A sequence with no cached token gets zeros.  The CTA of query
// head 0 also zeroes the sequence's stage-claim counter for the next call (the chunk kernel,
// the counter's only user, is complete here).
__global__ void __launch_bounds__(kDecCombineThreads)
    decode_combine_kernel(const __grid_constant__ DecPlan plan, const float *__restrict__ opart,
                          const float2 *__restrict__ mlpart, float *__restrict__ out, unsigned int *claims) {
  __shared__ __align__(16) float wo[kDecCombineWarps][128];
  __shared__ float2 wml[kDecCombineWarps];
  pdl_wait_and_release();                   // the chunk kernel's partials are complete and visible
  const int s = blockIdx.x / plan.hq, hh = blockIdx.x % plan.hq;
  if (hh == 0 && threadIdx.x == 0) claims[s] = 0u;
  const DecSeq &sq = plan.seq[s];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float m = -INFINITY, l = 0.f, o[4] = {0.f, 0.f, 0.f, 0.f};
  constexpr int kBatch = 10;                // chunk partials loaded before they are merged (one
                                            // round for up to 160 chunks)
  for (int c0 = warp; c0 < sq.nchunks; c0 += kDecCombineWarps * kBatch) {
    float2 ml[kBatch];
    float4 a[kBatch];
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const int cc = c0 + i * kDecCombineWarps;
      const int64_t idx = static_cast<int64_t>(sq.chunk_begin + cc) * plan.hq + hh;
      ml[i] = cc < sq.nchunks ? mlpart[idx] : make_float2(-INFINITY, 0.f);
      a[i] = cc < sq.nchunks ? *reinterpret_cast<const float4 *>(opart + idx * 128 + lane * 4)
                             : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int i = 0; i < kBatch; ++i) {
      const float o2[4] = {a[i].x, a[i].y, a[i].z, a[i].w};
      merge_state(m, l, o, ml[i].x, ml[i].y, o2);
    }
  }
  *reinterpret_cast<float4 *>(&wo[warp][lane * 4]) = make_float4(o[0], o[1], o[2], o[3]);
  if (lane == 0) wml[warp] = make_float2(m, l);
  __syncthreads();
  if (warp == 0) {
    float M = -INFINITY, L = 0.f, O[4] = {0.f, 0.f, 0.f, 0.f};
    for (int w = 0; w < kDecCombineWarps; ++w) {
      const float4 a = *reinterpret_cast<const float4 *>(&wo[w][lane * 4]);
      const float o2[4] = {a.x, a.y, a.z, a.w};
      merge_state(M, L, O, wml[w].x, wml[w].y, o2);
    }
    const float inv = L > 0.f ? 1.f / L : 0.f;
    *reinterpret_cast<float4 *>(out + (static_cast<int64_t>(s) * plan.hq + hh) * 128 + lane * 4) =
        make_float4(O[0] * inv, O[1] * inv, O[2] * inv, O[3] * inv);
  }
}

// The tensor-core chunk kernel takes Hkv = 2 or 4 with at most 8 query heads per KV head.
bool decode_tc_applies(int32_t hq, int32_t hkv) { return (hkv == 2 || hkv == 4) && hq / hkv <= kDecRows; }

// Keys per chunk: about one CTA per SM over the whole batch, whole 128-key tiles (a multiple of
// every stage size of both chunk kernels).
int decode_chunk_keys(int64_t total_tokens, int32_t hkv) {
  (void)hkv;
  const int64_t ctas = device_sm_count();
  int64_t c = (total_tokens + ctas - 1) / std::max<int64_t>(1, ctas);
  c = (c + 127) / 128 * 128;
  return static_cast<int>(std::min<int64_t>(std::max<int64_t>(c, 128), 1 << 20));
}

apack_status decode_validate(int32_t num_seqs, const int32_t *cu_seqlens_h, int32_t hq, int32_t hkv,
                             int64_t *total) {
  if (num_seqs < 0 || (num_seqs > 0 && !cu_seqlens_h)) return APACK_EINVAL;
  if (hq < 1 || hkv < 1 || hq % hkv != 0) return APACK_EINVAL;
  if (hq / hkv > kDecRows || hkv > 8 || kDecConsumers % hkv != 0) return APACK_EUNSUPPORTED;
  if (num_seqs > 0 && cu_seqlens_h[0] != 0) return APACK_EINVAL;
  for (int b = 0; b < num_seqs; ++b)
    if (cu_seqlens_h[b + 1] < cu_seqlens_h[b]) return APACK_EINVAL;
  *total = num_seqs > 0 ? cu_seqlens_h[num_seqs] : 0;
  return APACK_OK;
}

size_t up256(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

}  // namespace

}  // namespace apack

using namespace apack;

extern "C" {

apack_status apack_decode_workspace_size(int32_t num_seqs, const int32_t *cu_seqlens_h, int32_t num_q_heads,
                                         int32_t num_kv_heads, size_t *bytes) {
  if (!bytes) return APACK_EINVAL;
  int64_t total = 0;
  const apack_status st = decode_validate(num_seqs, cu_seqlens_h, num_q_heads, num_kv_heads, &total);
  if (st != APACK_OK) return st;
  const int chunk = decode_chunk_keys(total, num_kv_heads);
  int64_t chunks = 0;
  for (int b = 0; b < num_seqs; ++b) chunks += (cu_seqlens_h[b + 1] - cu_seqlens_h[b] + chunk - 1) / chunk;
  // device error word, chunk partials o [chunks][Hq][128] and (max, sum) [chunks][Hq], one
  // stage-claim counter per sequence
  *bytes = 256 + up256(static_cast<size_t>(chunks) * num_q_heads * 128 * sizeof(float)) +
           up256(static_cast<size_t>(chunks) * num_q_heads * sizeof(float2)) +
           up256(static_cast<size_t>(num_seqs) * sizeof(unsigned int));
  return APACK_OK;
}

apack_status apack_decode_attention(int32_t num_seqs, const int32_t *cu_seqlens_h, const void *q, const void *k,
                                    const void *v, int64_t kv_token_stride, int32_t num_q_heads,
                                    int32_t num_kv_heads, float *out, void *ws, size_t ws_bytes, void *stream) {
  int64_t total = 0;
  apack_status st = decode_validate(num_seqs, cu_seqlens_h, num_q_heads, num_kv_heads, &total);
  if (st != APACK_OK) return st;
  if (num_seqs == 0) return APACK_OK;
  if (!q || !k || !v || !out || !ws) return APACK_EINVAL;
  if (in_host_memory(k) || in_host_memory(v)) return APACK_EINVAL;   // read by TMA / bulk copies
  if ((reinterpret_cast<uintptr_t>(q) & 7) || (reinterpret_cast<uintptr_t>(k) & 15) ||
      (reinterpret_cast<uintptr_t>(v) & 15) || (reinterpret_cast<uintptr_t>(out) & 15) ||
      (reinterpret_cast<uintptr_t>(ws) & 255) || (kv_token_stride & 15) ||
      kv_token_stride < static_cast<int64_t>(num_kv_heads) * 256)
    return APACK_EINVAL;
  size_t need = 0;
  apack_decode_workspace_size(num_seqs, cu_seqlens_h, num_q_heads, num_kv_heads, &need);
  if (ws_bytes < need) return APACK_EWORKSPACE;
  const int chunk = decode_chunk_keys(total, num_kv_heads);
  int64_t chunks_all = 0;
  for (int b = 0; b < num_seqs; ++b) chunks_all += (cu_seqlens_h[b + 1] - cu_seqlens_h[b] + chunk - 1) / chunk;
  DeviceError *err = static_cast<DeviceError *>(ws);
  float *opart = reinterpret_cast<float *>(static_cast<uint8_t *>(ws) + 256);
  float2 *mlpart = reinterpret_cast<float2 *>(static_cast<uint8_t *>(ws) + 256 +
                                              up256(static_cast<size_t>(chunks_all) * num_q_heads * 128 * sizeof(float)));
  unsigned int *claims = reinterpret_cast<unsigned int *>(
      reinterpret_cast<uint8_t *>(mlpart) + up256(static_cast<size_t>(chunks_all) * num_q_heads * sizeof(float2)));
  static std::atomic<uint64_t> attr_done{0};
  if (once_per_device(attr_done, [] {
        return cudaFuncSetAttribute(decode_chunk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(kDecSmem));
      }) != cudaSuccess)
    return APACK_ECUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint16_t *q16 = static_cast<const uint16_t *>(q);
  const bool tc = decode_tc_applies(num_q_heads, num_kv_heads) && total > 0;
  CUtensorMap kmap, vmap;
  if (tc && (!make_kv_tile_map(&kmap, k, num_kv_heads, total, kv_token_stride, 128) ||
             !make_kv_tile_map(&vmap, v, num_kv_heads, total, kv_token_stride, 128)))
    return APACK_ECUDA;
  int64_t chunk_base = 0;
  for (int s0 = 0; s0 < num_seqs; s0 += kSeqsPerLaunch) {
    const int ns = std::min(num_seqs - s0, kSeqsPerLaunch);
    DecPlan P{};
    P.nseq = ns;
    P.hq = num_q_heads;
    P.hkv = num_kv_heads;
    P.group = num_q_heads / num_kv_heads;
    P.chunk = chunk;                    // whole 128-key tiles
    P.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(APACK_HEAD_DIM)));
    int chunks = 0;
    for (int i = 0; i < ns; ++i) {
      DecSeq &d = P.seq[i];
      d.t0 = cu_seqlens_h[s0 + i];
      d.len = cu_seqlens_h[s0 + i + 1] - d.t0;
      d.chunk_begin = chunks;
      d.nchunks = (d.len + chunk - 1) / chunk;
      chunks += d.nchunks;
    }
    P.total_chunks = chunks;
    float *op = opart + chunk_base * num_q_heads * 128;
    float2 *mp = mlpart + chunk_base * num_q_heads;
    const uint16_t *qs = q16 + static_cast<int64_t>(s0) * num_q_heads * 128;
    if (chunks > 0) {
      if (tc) {
        if (check_cuda(launch_decode_tc(chunks, s, kmap, vmap, P, qs, op, mp, claims + s0, err)) != APACK_OK)
          return APACK_ECUDA;
      } else {
        decode_chunk_kernel<<<chunks, kDecThreads, kDecSmem, s>>>(P, qs, static_cast<const uint8_t *>(k),
                                                                  static_cast<const uint8_t *>(v), kv_token_stride,
                                                                  op, mp, err);
        if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
      }
      count_launches(1);
    }
    // programmatic dependent launch: the combine's CTAs are scheduled while the chunk kernel
    // drains and wait (griddepcontrol.wait) for its completion before reading the partials
    if (check_cuda(launch_pdl(decode_combine_kernel, dim3(ns * num_q_heads), dim3(kDecCombineThreads), 0, s, P,
                              static_cast<const float *>(op), static_cast<const float2 *>(mp),
                              out + static_cast<int64_t>(s0) * num_q_heads * 128, claims + s0)) != APACK_OK)
      return APACK_ECUDA;
    count_launches(1);
    chunk_base += chunks;
  }
  return APACK_OK;
}

}  // extern "C"
