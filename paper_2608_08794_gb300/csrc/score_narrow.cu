// score_narrow.cu -- relevance scores of Eq. inner_score (Sec. 3.2) when each KV head group
// has few query rows: the paper's own setting scores with the last query token only
// (Table S-hparams), i.e. G = Hq/Hkv rows per group (7 for the 7B model).
//
// With so few rows the step is bound by reading K once, so the logits are computed once and
// kept: three launches.
//   logits kernel:  log2-domain logits x * log2(e)/sqrt(D) of every (logit row, key), stored per
//                   logit row with a row stride padded to 64 keys, and per CTA the (max, sum of
//                   exp2) of every logit row over its multimodal keys.  Two variants:
//                   * Hkv = 2 or 4 with at most 8 rows per head group: the tcgen05 kernel of
//                     score_narrow_tc.cu (keys as M = 128, the group's rows as N = 16);
//                   * other shapes: one thread per key reads its whole token row and dots it
//                     with the group's query rows held in shared memory;
//   merge kernel:   per logit row, one block combines the CTA partials into lse2;
//   final kernel:   one thread per key sums exp2(logit - lse2) over all logit rows
//                   in a fixed order and scales by 1/(Hq n_q).
// The logits of the 10-minute 7B sequence with one query row take 15 MB and stay
// in L2 between the first and the last kernel.
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "narrow_plan.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kThreads = 256;          // keys per CTA (general logits kernel, final kernel)
constexpr int kWarps = kThreads / 32;
constexpr int kRows8Tokens = 64;       // lower bound of the tensor-core kernel's key chunk (sizes partials)
constexpr int kLogitPad = 64;          // logit row stride: the key count rounded up to this

__device__ __forceinline__ bool is_mm(uint8_t m) { return m == APACK_MOD_AUDIO || m == APACK_MOD_VISUAL; }

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

__device__ __forceinline__ void bf16x8_to_f32(const uint4 &v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

// RG = compile-time upper bound of the rows of one KV head group (G * n_q <= RG).
template <int RG>
__global__ void __launch_bounds__(kThreads)
    score_narrow_logits_kernel(const __grid_constant__ NarrowPlan plan, const uint16_t *__restrict__ q,
                               const uint8_t *__restrict__ k, int64_t k_stride, const uint8_t *__restrict__ modality,
                               float *__restrict__ logits, float2 *__restrict__ part) {
  pdl_wait_and_release();
  extern __shared__ __align__(16) float smem_f[];
  const int s = find_unit_seq(plan, blockIdx.x);
  const NSeq &sq = plan.seq[s];
  const int R = sq.rows;
  float *qs = smem_f;                                                  // [R][128]
  float2 *wpart = reinterpret_cast<float2 *>(smem_f + R * 128);       // [kWarps][R]
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int kt = blockIdx.x - sq.unit_begin;
  const int key = sq.t0 + kt * kThreads + tid;
  const bool in = key < sq.t0 + sq.len;
  const bool mm = in && is_mm(modality[key]);
  // query rows of the sequence: logit row rho = token * Hq + head (the order of Q in memory)
  for (int i = tid; i < R * 128; i += kThreads)
    qs[i] = __uint_as_float(static_cast<uint32_t>(q[static_cast<int64_t>(sq.q_off) * plan.hq * 128 + i]) << 16);
  __syncthreads();
  const int G = plan.group, rg = G * sq.n_q;
  const uint8_t *krow = k + static_cast<int64_t>(in ? key : sq.t0) * k_stride;
  const int64_t lbase = sq.logit_base + (key - sq.t0);
  for (int g = 0; g < plan.hkv; ++g) {
    float acc[RG];
    int qoff[RG];                      // logit row rho = token * Hq + g * G + j, as an offset into qs
#pragma unroll
    for (int l = 0; l < RG; ++l) {
      acc[l] = 0.f;
      qoff[l] = l < rg ? ((l / G) * plan.hq + g * G + (l % G)) * 128 : 0;
    }
    const uint4 *kg = reinterpret_cast<const uint4 *>(krow + g * 256);
#pragma unroll 4
    for (int c = 0; c < 16; ++c) {
      float kf[8];
      bf16x8_to_f32(in ? __ldg(kg + c) : make_uint4(0, 0, 0, 0), kf);
#pragma unroll
      for (int l = 0; l < RG; ++l) {
        if (l < rg) {
          const float4 qa = *reinterpret_cast<const float4 *>(qs + qoff[l] + c * 8);
          const float4 qb = *reinterpret_cast<const float4 *>(qs + qoff[l] + c * 8 + 4);
          acc[l] = fmaf(kf[0], qa.x, acc[l]);
          acc[l] = fmaf(kf[1], qa.y, acc[l]);
          acc[l] = fmaf(kf[2], qa.z, acc[l]);
          acc[l] = fmaf(kf[3], qa.w, acc[l]);
          acc[l] = fmaf(kf[4], qb.x, acc[l]);
          acc[l] = fmaf(kf[5], qb.y, acc[l]);
          acc[l] = fmaf(kf[6], qb.z, acc[l]);
          acc[l] = fmaf(kf[7], qb.w, acc[l]);
        }
      }
    }
#pragma unroll
    for (int l = 0; l < RG; ++l) {
      if (l < rg) {
        const int rho = qoff[l] / 128;
        const float y = acc[l] * plan.scale2;
        if (in) logits[lbase + static_cast<int64_t>(rho) * sq.lstride] = y;
        // this warp's (max, sum of exp2) of the row over the keys in its denominator: the
        // multimodal keys, or (causal rows) every key up to the row's own position
        const bool use = plan.causal ? (in && key - sq.t0 <= sq.q_pos + l / G) : mm;
        const float wm = warp_max(use ? y : -INFINITY);
        const float ws = warp_sum(use && wm != -INFINITY ? ex2_approx(y - wm) : 0.f);
        if (lane == 0) wpart[warp * R + rho] = make_float2(wm, ws);
      }
    }
  }
  __syncthreads();
  for (int rho = tid; rho < R; rho += kThreads) {
    float m = -INFINITY;
    for (int w = 0; w < kWarps; ++w) m = fmaxf(m, wpart[w * R + rho].x);
    float sum = 0.f;
    if (m != -INFINITY)
      for (int w = 0; w < kWarps; ++w) {
        const float2 v = wpart[w * R + rho];
        if (v.x != -INFINITY) sum += v.y * ex2_approx(v.x - m);
      }
    part[sq.part_base + static_cast<int64_t>(kt) * R + rho] = make_float2(m, sum);
  }
}

// One block per (sequence, logit row): lse2 over the CTA partials.  Each thread
// folds a fixed stride of partials, then a fixed-shape tree combines the
// threads: the order never depends on timing, so lse2 is deterministic.
__global__ void __launch_bounds__(kThreads)
    score_narrow_merge_kernel(const __grid_constant__ NarrowPlan plan, const float2 *__restrict__ part,
                              float *__restrict__ lse2) {
  pdl_wait_and_release();
  __shared__ float red[kWarps];
  __shared__ float mshared;
  const int64_t e = blockIdx.x;
  int s = 0;
  int64_t acc = 0;
  while (s + 1 < plan.nseq && acc + plan.seq[s].rows <= e) acc += plan.seq[s++].rows;
  const NSeq &sq = plan.seq[s];
  const int rho = static_cast<int>(e - acc);
  const int ctas = sq.nparts;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  // up to kHold partials per thread are loaded once, together, and kept for the sum
  constexpr int kHold = 8;
  const bool held = ctas <= kHold * kThreads;
  float2 v[kHold];
  float m = -INFINITY;
  if (held) {
#pragma unroll
    for (int i = 0; i < kHold; ++i) {
      const int c = tid + i * kThreads;
      v[i] = c < ctas ? part[sq.part_base + static_cast<int64_t>(c) * sq.rows + rho] : make_float2(-INFINITY, 0.f);
      m = fmaxf(m, v[i].x);
    }
  } else {
    for (int c = tid; c < ctas; c += kThreads) m = fmaxf(m, part[sq.part_base + static_cast<int64_t>(c) * sq.rows + rho].x);
  }
  m = warp_max(m);
  if (lane == 0) red[warp] = m;
  __syncthreads();
  if (tid == 0) {
    float mm = -INFINITY;
    for (int w = 0; w < kWarps; ++w) mm = fmaxf(mm, red[w]);
    mshared = mm;
  }
  __syncthreads();
  m = mshared;
  float sum = 0.f;
  if (m != -INFINITY) {
    if (held) {
#pragma unroll
      for (int i = 0; i < kHold; ++i)   // the same partials in the same order as the loop below
        if (v[i].x != -INFINITY) sum += v[i].y * exp2f(v[i].x - m);
    } else {
      for (int c = tid; c < ctas; c += kThreads) {
        const float2 w = part[sq.part_base + static_cast<int64_t>(c) * sq.rows + rho];
        if (w.x != -INFINITY) sum += w.y * exp2f(w.x - m);
      }
    }
  }
  sum = warp_sum(sum);
  __syncthreads();
  if (lane == 0) red[warp] = sum;
  __syncthreads();
  if (tid == 0) {
    float tot = 0.f;
    for (int w = 0; w < kWarps; ++w) tot += red[w];
    // no multimodal key: nothing is scored in this sequence
    lse2[sq.lse_base + rho] = m == -INFINITY ? INFINITY : m + log2f(tot);
  }
}

// One thread per key: I = sum over logit rows of exp2(logit - lse2) / (Hq n_q).
__global__ void __launch_bounds__(kThreads)
    score_narrow_final_kernel(const __grid_constant__ NarrowPlan plan, const uint8_t *__restrict__ modality,
                              const float *__restrict__ logits, const float *__restrict__ lse2,
                              float *__restrict__ scores) {
  pdl_wait_and_release();
  extern __shared__ __align__(16) float ls[];
  const int s = find_unit_seq(plan, blockIdx.x);
  const NSeq &sq = plan.seq[s];
  const int R = sq.rows;
  const int kt = blockIdx.x - sq.unit_begin;
  const int key = sq.t0 + kt * kThreads + threadIdx.x;
  const bool in = key < sq.t0 + sq.len;
  const float *lp = logits + sq.logit_base + (key - sq.t0);
  // the key's own loads (modality, and up to 32 rows' logits) are issued before the normalisers
  // arrive: one round trip for all of them
  const uint8_t mod = in ? modality[key] : static_cast<uint8_t>(0);
  float raw[32];
  if (R <= 32) {
#pragma unroll
    for (int u = 0; u < 32; ++u) raw[u] = (in && u < R) ? lp[static_cast<int64_t>(u) * sq.lstride] : 0.f;
  }
  for (int i = threadIdx.x; i < R; i += kThreads) ls[i] = lse2[sq.lse_base + i];
  __syncthreads();
  if (!in) return;
  float out = 0.f;
  if (sq.n_q > 0 && is_mm(mod)) {
    // eight independent sums, the loads of a block of 8 rows issued together
    float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    // causal rows: logit row rho = token * Hq + head sees this key when token >= key - q_pos
    const int rho_min = plan.causal ? max(0, key - sq.t0 - sq.q_pos) * plan.hq : 0;
    if (R <= 32) {
      // all rows (the paper's one query token: R = Hq)
      float x[32];
#pragma unroll
      for (int u = 0; u < 32; ++u) x[u] = (u < R && u >= rho_min) ? raw[u] - ls[u] : -INFINITY;
#pragma unroll
      for (int u = 0; u < 32; ++u) a[u & 7] += ex2_approx(x[u]);
    } else {
      for (int r0 = 0; r0 < R; r0 += 8) {
        float x[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          x[u] = (r0 + u < R && r0 + u >= rho_min) ? lp[static_cast<int64_t>(r0 + u) * sq.lstride] - ls[r0 + u]
                                                   : -INFINITY;
#pragma unroll
        for (int u = 0; u < 8; ++u) a[u] += ex2_approx(x[u]);
      }
    }
    out = (((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]))) / static_cast<float>(plan.hq * sq.n_q);
  }
  scores[key] = out;
}

template <int RG>
cudaError_t launch_logits(int grid, size_t smem, cudaStream_t stream, const NarrowPlan &P, const uint16_t *q,
                          const uint8_t *k, int64_t k_stride, const uint8_t *modality, float *logits, float2 *part) {
  static std::atomic<uint64_t> attr{0};
  const cudaError_t e = once_per_device(attr, [] {
    return cudaFuncSetAttribute(score_narrow_logits_kernel<RG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                160 * 1024);
  });
  if (e != cudaSuccess) return e;
  return launch_pdl(score_narrow_logits_kernel<RG>, dim3(grid), dim3(kThreads), smem, stream, P, q, k, k_stride,
                    modality, logits, part);
}

}  // namespace

bool narrow_score_applies(const apack_seqs *s) {
  const int G = s->num_q_heads / s->num_kv_heads;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int nq = s->cu_qlens_h[b + 1] - s->cu_qlens_h[b];
    if (G * nq > kNarrowGroupRows || s->num_q_heads * nq > kNarrowRows) return false;
  }
  return true;
}

void narrow_layout(const apack_seqs *s, size_t *logit_floats, size_t *part_float2s, size_t *lse_floats) {
  size_t lf = 0, pf = 0, ef = 0;
  for (int b = 0; b < s->num_seqs; ++b) {
    const int64_t len = s->cu_seqlens_h[b + 1] - s->cu_seqlens_h[b];
    const int64_t R = static_cast<int64_t>(s->num_q_heads) * (s->cu_qlens_h[b + 1] - s->cu_qlens_h[b]);
    lf += static_cast<size_t>(R * ((len + kLogitPad - 1) / kLogitPad * kLogitPad));
    pf += static_cast<size_t>(R * ((len + kRows8Tokens - 1) / kRows8Tokens));   // enough for either kernel
    ef += static_cast<size_t>(R);
  }
  *logit_floats = lf;
  *part_float2s = pf;
  *lse_floats = ef;
}

apack_status run_score_narrow(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                              float *scores, void *ws, cudaStream_t stream) {
  const WsLayout L = workspace_layout(seqs);
  uint8_t *wsb = static_cast<uint8_t *>(ws);
  float *logits = reinterpret_cast<float *>(wsb + L.nlog_off);
  float2 *part = reinterpret_cast<float2 *>(wsb + L.npart_off);
  float *lse2 = reinterpret_cast<float *>(wsb + L.nlse_off);
  const int B = seqs->num_seqs;
  const int hq = seqs->num_q_heads, hkv = seqs->num_kv_heads, G = hq / hkv;
  int64_t logit_base = 0, part_base = 0, lse_base = 0;
  for (int s0 = 0; s0 < B; s0 += kSeqsPerLaunch) {
    const int ns = (B - s0 < kSeqsPerLaunch) ? (B - s0) : kSeqsPerLaunch;
    NarrowPlan P{};
    P.nseq = ns;
    P.hq = hq;
    P.hkv = hkv;
    P.group = G;
    P.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(APACK_HEAD_DIM)));
    P.causal = seqs->softmax_domain == APACK_SOFTMAX_CAUSAL_ROW;
    // tensor-core logits kernel: Hkv = 2 or 4, at most 8 rows per head group
    int max_rg = 0;
    for (int i = 0; i < ns; ++i) {
      const int nq = seqs->cu_qlens_h[s0 + i + 1] - seqs->cu_qlens_h[s0 + i];
      max_rg = G * nq > max_rg ? G * nq : max_rg;
    }
    const bool rows8 = (hkv == 2 || hkv == 4) && max_rg <= 8;
    // its chunk: about one CTA per SM over this launch's keys, whole 128-key tiles
    int64_t launch_tokens = 0;
    for (int i = 0; i < ns; ++i) launch_tokens += seqs->cu_seqlens_h[s0 + i + 1] - seqs->cu_seqlens_h[s0 + i];
    const int64_t stage_tok = 128;     // chunks are whole 128-key tensor-core tiles
    const int64_t sms = device_sm_count();
    int64_t chunk = (launch_tokens + sms - 1) / sms;
    chunk = std::max<int64_t>(stage_tok, (chunk + stage_tok - 1) / stage_tok * stage_tok);
    P.chunk = static_cast<int32_t>(std::min<int64_t>(chunk, 1 << 24));
    int units = 0, units8 = 0, max_rows = 0;
    int64_t rows_all = 0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      NSeq &sq = P.seq[i];
      sq.t0 = seqs->cu_seqlens_h[b];
      sq.len = seqs->cu_seqlens_h[b + 1] - sq.t0;
      sq.q_off = seqs->cu_qlens_h[b];
      sq.n_q = seqs->cu_qlens_h[b + 1] - sq.q_off;
      sq.rows = hq * sq.n_q;
      sq.q_pos = query_position(seqs, b);
      sq.unit_begin = units;
      sq.unit8_begin = units8;
      sq.lstride = (sq.len + kLogitPad - 1) / kLogitPad * kLogitPad;
      sq.logit_base = logit_base;
      sq.part_base = part_base;
      sq.lse_base = lse_base;
      const int ctas = (sq.len + kThreads - 1) / kThreads;
      const int ctas8 = (sq.len + P.chunk - 1) / P.chunk;   // <= (len + 63) / 64: fits the workspace
      sq.nparts = rows8 ? ctas8 : ctas;
      units += ctas;
      units8 += ctas8;
      logit_base += static_cast<int64_t>(sq.rows) * sq.lstride;
      part_base += static_cast<int64_t>(sq.rows) * ctas8;
      lse_base += sq.rows;
      rows_all += sq.rows;
      max_rows = sq.rows > max_rows ? sq.rows : max_rows;
    }
    P.total_units = units;
    P.total_units8 = units8;
    if (units == 0) continue;
    cudaError_t e;
    const uint16_t *q16 = static_cast<const uint16_t *>(q);
    const uint8_t *k8 = static_cast<const uint8_t *>(k);
    if (rows8) {
      DeviceError *err = reinterpret_cast<DeviceError *>(wsb + L.err_off);
      CUtensorMap kmap;
      if (!make_kv_tile_map(&kmap, k, hkv, seqs->cu_seqlens_h[B], k_token_stride, 128)) return APACK_ECUDA;
      e = launch_narrow_tc(units8, stream, kmap, P, q16, seqs->modality, logits, part, err);
    } else {
      const size_t smem = static_cast<size_t>(max_rows) * 128 * sizeof(float) +
                          static_cast<size_t>(kWarps) * max_rows * sizeof(float2);
      if (max_rg <= 8)
        e = launch_logits<8>(units, smem, stream, P, q16, k8, k_token_stride, seqs->modality, logits, part);
      else if (max_rg <= 16)
        e = launch_logits<16>(units, smem, stream, P, q16, k8, k_token_stride, seqs->modality, logits, part);
      else
        e = launch_logits<32>(units, smem, stream, P, q16, k8, k_token_stride, seqs->modality, logits, part);
    }
    count_launches(1);
    if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
    if (rows_all > 0) {
      if (check_cuda(launch_pdl(score_narrow_merge_kernel, dim3(static_cast<unsigned>(rows_all)), dim3(kThreads), 0,
                                stream, P, part, lse2)) != APACK_OK)
        return APACK_ECUDA;
      count_launches(1);
    }
    if (check_cuda(launch_pdl(score_narrow_final_kernel, dim3(units), dim3(kThreads),
                              static_cast<size_t>(max_rows) * sizeof(float), stream, P, seqs->modality, logits, lse2,
                              scores)) != APACK_OK)
      return APACK_ECUDA;
    count_launches(1);
  }
  return APACK_OK;
}

}  // namespace apack
