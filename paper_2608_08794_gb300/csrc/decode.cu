// decode.cu -- attention of one decode token over a (compacted) KV cache: the cost the
// inner-LLM pruning shortens for every autoregressive step (Sec. 3.2, last sentence;
// App. G, decoding throughput).
//
//   out[b, h] = sum_j softmax_j(q[b, h] . k[j, g(h)] / sqrt(128)) v[j, g(h)],
//   g(h) = h / (Hq / Hkv), j over every cached token of sequence b.
//
// Split-KV in two launches:
//   chunk kernel:   one CTA per (sequence, chunk of keys), 8 warps; warp w works on KV
//                   head w % Hkv and a contiguous run of the chunk's keys; lane l owns
//                   features [4l, 4l + 4) of that head for all G <= 8 query rows of the
//                   head group.  Per 8 keys: logits by a reduce-scatter of the 8 row
//                   partials over the warp (the lane's query rows are stored in an
//                   order that makes every step a plain shuffle and add), online max
//                   and sum per row, probabilities handed to all lanes through shared
//                   memory, P.V accumulated in registers.  Warps of the same head merge
//                   in shared memory; the CTA writes (max, sum, o[128]) per query head.
//   combine kernel: one CTA per (sequence, query head) merges the chunks in order.
// K and V are read once: the chunk kernel is HBM-bound.  All merges run in a fixed
// order, so the output is deterministic.
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kDecRows = 8;              // query rows per KV head group (G <= 8)
constexpr int kDecCombineThreads = 512;
constexpr int kDecCombineWarps = kDecCombineThreads / 32;

struct DecSeq {
  int32_t t0, len;
  int32_t chunk_begin, nchunks;
};

struct DecPlan {
  int32_t nseq, hq, hkv, group, chunk;   // chunk: keys per CTA, a multiple of 64
  int32_t total_chunks;
  float scale2;                          // log2(e) / sqrt(128)
  DecSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int find_chunk_seq(const DecPlan &p, int c) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].chunk_begin <= c) ++s;
  return s;
}

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
__global__ void __launch_bounds__(kDecThreads, 2)
    decode_chunk_kernel(const __grid_constant__ DecPlan plan, const uint16_t *__restrict__ q,
                        const uint8_t *__restrict__ k, const uint8_t *__restrict__ v, int64_t kv_stride,
                        float *__restrict__ opart, float2 *__restrict__ mlpart) {
  __shared__ __align__(16) float ps[kDecWarps][8][kDecRows];   // [warp][key][row] probabilities
  __shared__ __align__(16) float sc[kDecWarps][kDecRows];      // [warp][row] rescale factors
  __shared__ __align__(16) float wo[kDecWarps][kDecRows][128]; // per warp o, for the head merge
  __shared__ float2 wml[kDecWarps][kDecRows];                  // per warp (max, sum) per row
  const int c = blockIdx.x;
  const int s = find_chunk_seq(plan, c);
  const DecSeq &sq = plan.seq[s];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int G = plan.group, hkv = plan.hkv;
  const int h = warp % hkv, stream = warp / hkv, nstreams = kDecWarps / hkv;
  // keys of this warp: a contiguous run of the chunk
  const int cbeg = (c - sq.chunk_begin) * plan.chunk;
  const int per = plan.chunk / nstreams;
  const int tb = cbeg + stream * per;
  const int te = min(sq.len, tb + per);
  // query rows of the group, lane-permuted: slot j holds row j ^ cl
  const int cl = (lane >> 2) & 7;
  float qf[kDecRows][4];
  const uint16_t *qg = q + (static_cast<int64_t>(s) * plan.hq + h * G) * 128 + lane * 4;
#pragma unroll
  for (int j = 0; j < kDecRows; ++j) {
    const int row = j ^ cl;
    uint2 w = make_uint2(0, 0);
    if (row < G) w = __ldg(reinterpret_cast<const uint2 *>(qg + row * 128));
    bf16x4_to_f32(w, qf[j]);
  }
  // after the reduce-scatter this lane holds the logit of row cl
  float o[kDecRows][4];
#pragma unroll
  for (int j = 0; j < kDecRows; ++j) o[j][0] = o[j][1] = o[j][2] = o[j][3] = 0.f;
  float m_own = -INFINITY, l_own = 0.f;
  const uint8_t *kb = k + static_cast<int64_t>(sq.t0) * kv_stride + h * 256 + lane * 8;
  const uint8_t *vb = v + static_cast<int64_t>(sq.t0) * kv_stride + h * 256 + lane * 8;
#pragma unroll 1
  for (int t0 = tb; t0 < te; t0 += 8) {
    uint2 kr[8], vr[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const bool ok = t0 + i < te;
      kr[i] = ok ? __ldg(reinterpret_cast<const uint2 *>(kb + static_cast<int64_t>(t0 + i) * kv_stride))
                 : make_uint2(0, 0);
      vr[i] = ok ? __ldg(reinterpret_cast<const uint2 *>(vb + static_cast<int64_t>(t0 + i) * kv_stride))
                 : make_uint2(0, 0);
    }
    float x[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float kf[4];
      bf16x4_to_f32(kr[i], kf);
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
      x[i] = t0 + i < te ? acc[0] * plan.scale2 : -INFINITY;
    }
    // online softmax of row cl over these keys (key t0 is always valid)
    float cm = x[0];
#pragma unroll
    for (int i = 1; i < 8; ++i) cm = fmaxf(cm, x[i]);
    const float mn = fmaxf(m_own, cm);
    const float scale = ex2_approx(m_own - mn);
    float psum = 0.f;
    __syncwarp();
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float p = ex2_approx(x[i] - mn);
      psum += p;
      ps[warp][i][cl] = p;               // the four lanes of a row write the same value
    }
    sc[warp][cl] = scale;
    l_own = l_own * scale + psum;
    m_own = mn;
    __syncwarp();
    {
      const float4 sa = *reinterpret_cast<const float4 *>(&sc[warp][0]);
      const float4 sb = *reinterpret_cast<const float4 *>(&sc[warp][4]);
      const float sr[8] = {sa.x, sa.y, sa.z, sa.w, sb.x, sb.y, sb.z, sb.w};
#pragma unroll
      for (int j = 0; j < kDecRows; ++j)
#pragma unroll
        for (int e = 0; e < 4; ++e) o[j][e] *= sr[j];
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      float vf[4];
      bf16x4_to_f32(vr[i], vf);
      const float4 pa = *reinterpret_cast<const float4 *>(&ps[warp][i][0]);
      const float4 pb = *reinterpret_cast<const float4 *>(&ps[warp][i][4]);
      const float pr[8] = {pa.x, pa.y, pa.z, pa.w, pb.x, pb.y, pb.z, pb.w};
#pragma unroll
      for (int j = 0; j < kDecRows; j += 2)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float2 r = ffma2(make_float2(pr[j], pr[j + 1]), make_float2(vf[e], vf[e]),
                                 make_float2(o[j][e], o[j + 1][e]));
          o[j][e] = r.x;
          o[j + 1][e] = r.y;
        }
    }
  }
  // merge the warps of each head in stream order, then write the chunk's partials
#pragma unroll
  for (int j = 0; j < kDecRows; ++j)
    *reinterpret_cast<float4 *>(&wo[warp][j][lane * 4]) = make_float4(o[j][0], o[j][1], o[j][2], o[j][3]);
  if ((lane & 3) == 0) wml[warp][cl] = make_float2(m_own, l_own);
  __syncthreads();
  if (stream == 0) {
    // this warp (stream 0 of head h) folds in streams 1.. of the same head
    for (int st = 1; st < nstreams; ++st) {
      const int w2 = st * hkv + h;
#pragma unroll
      for (int j = 0; j < kDecRows; ++j) {
        float m1 = wml[warp][j].x, l1 = wml[warp][j].y;
        const float2 ml2 = wml[w2][j];
        float o1[4], o2[4];
        const float4 a = *reinterpret_cast<const float4 *>(&wo[warp][j][lane * 4]);
        const float4 b = *reinterpret_cast<const float4 *>(&wo[w2][j][lane * 4]);
        o1[0] = a.x; o1[1] = a.y; o1[2] = a.z; o1[3] = a.w;
        o2[0] = b.x; o2[1] = b.y; o2[2] = b.z; o2[3] = b.w;
        merge_state(m1, l1, o1, ml2.x, ml2.y, o2);
        *reinterpret_cast<float4 *>(&wo[warp][j][lane * 4]) = make_float4(o1[0], o1[1], o1[2], o1[3]);
        __syncwarp();
        if (lane == 0) wml[warp][j] = make_float2(m1, l1);
        __syncwarp();
      }
    }
    for (int j = 0; j < G; ++j) {
      const int64_t hq_idx = static_cast<int64_t>(c) * plan.hq + h * G + j;
      *reinterpret_cast<float4 *>(opart + hq_idx * 128 + lane * 4) =
          *reinterpret_cast<const float4 *>(&wo[warp][j][lane * 4]);
      if (lane == 0) mlpart[hq_idx] = wml[warp][j];
    }
  }
}

// One CTA per (sequence, query head): merge the sequence's chunks.  Warp w folds chunks
// w, w + 16, w + 32, ... in that order (lane: features [4 lane, 4 lane + 4)); the warps
// then merge in warp order.  A sequence with no cached token gets zeros.
__global__ void __launch_bounds__(kDecCombineThreads)
    decode_combine_kernel(const __grid_constant__ DecPlan plan, const float *__restrict__ opart,
                          const float2 *__restrict__ mlpart, float *__restrict__ out) {
  __shared__ __align__(16) float wo[kDecCombineWarps][128];
  __shared__ float2 wml[kDecCombineWarps];
  const int s = blockIdx.x / plan.hq, hh = blockIdx.x % plan.hq;
  const DecSeq &sq = plan.seq[s];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float m = -INFINITY, l = 0.f, o[4] = {0.f, 0.f, 0.f, 0.f};
  constexpr int kBatch = 4;                 // chunk partials loaded before they are merged
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

// Keys per chunk: about two CTAs per SM over the whole batch, a multiple of 64.
int decode_chunk_keys(int64_t total_tokens) {
  const int64_t ctas = 2 * static_cast<int64_t>(device_sm_count());
  int64_t c = (total_tokens + ctas - 1) / std::max<int64_t>(1, ctas);
  c = (c + 63) / 64 * 64;
  return static_cast<int>(std::min<int64_t>(std::max<int64_t>(c, 64), 1 << 16));
}

apack_status decode_validate(int32_t num_seqs, const int32_t *cu_seqlens_h, int32_t hq, int32_t hkv,
                             int64_t *total) {
  if (num_seqs < 0 || (num_seqs > 0 && !cu_seqlens_h)) return APACK_EINVAL;
  if (hq < 1 || hkv < 1 || hq % hkv != 0) return APACK_EINVAL;
  if (hq / hkv > kDecRows || kDecWarps % hkv != 0) return APACK_EUNSUPPORTED;
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
  const int chunk = decode_chunk_keys(total);
  int64_t chunks = 0;
  for (int b = 0; b < num_seqs; ++b) chunks += (cu_seqlens_h[b + 1] - cu_seqlens_h[b] + chunk - 1) / chunk;
  *bytes = up256(static_cast<size_t>(chunks) * num_q_heads * 128 * sizeof(float)) +
           up256(static_cast<size_t>(chunks) * num_q_heads * sizeof(float2));
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
  if ((reinterpret_cast<uintptr_t>(q) & 7) || (reinterpret_cast<uintptr_t>(k) & 7) ||
      (reinterpret_cast<uintptr_t>(v) & 7) || (reinterpret_cast<uintptr_t>(out) & 15) ||
      (reinterpret_cast<uintptr_t>(ws) & 255) || (kv_token_stride & 7) ||
      kv_token_stride < static_cast<int64_t>(num_kv_heads) * 256)
    return APACK_EINVAL;
  size_t need = 0;
  apack_decode_workspace_size(num_seqs, cu_seqlens_h, num_q_heads, num_kv_heads, &need);
  if (ws_bytes < need) return APACK_EWORKSPACE;
  const int chunk = decode_chunk_keys(total);
  int64_t chunks_all = 0;
  for (int b = 0; b < num_seqs; ++b) chunks_all += (cu_seqlens_h[b + 1] - cu_seqlens_h[b] + chunk - 1) / chunk;
  float *opart = static_cast<float *>(ws);
  float2 *mlpart = reinterpret_cast<float2 *>(static_cast<uint8_t *>(ws) +
                                              up256(static_cast<size_t>(chunks_all) * num_q_heads * 128 * sizeof(float)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint16_t *q16 = static_cast<const uint16_t *>(q);
  int64_t chunk_base = 0;
  for (int s0 = 0; s0 < num_seqs; s0 += kSeqsPerLaunch) {
    const int ns = std::min(num_seqs - s0, kSeqsPerLaunch);
    DecPlan P{};
    P.nseq = ns;
    P.hq = num_q_heads;
    P.hkv = num_kv_heads;
    P.group = num_q_heads / num_kv_heads;
    P.chunk = chunk;
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
      decode_chunk_kernel<<<chunks, kDecThreads, 0, s>>>(P, qs, static_cast<const uint8_t *>(k),
                                                         static_cast<const uint8_t *>(v), kv_token_stride, op, mp);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    decode_combine_kernel<<<ns * num_q_heads, kDecCombineThreads, 0, s>>>(
        P, op, mp, out + static_cast<int64_t>(s0) * num_q_heads * 128);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    chunk_base += chunks;
  }
  return APACK_OK;
}

}  // extern "C"
