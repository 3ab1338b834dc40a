// score_narrow.cu -- relevance scores of Eq. inner_score (Sec. 3.2) when each KV head group
// has few query rows: the paper's own setting scores with the last query token only
// (Table S-hparams), i.e. G = Hq/Hkv rows per group (7 for the 7B model).
//
// With so few rows the step is bound by reading K from HBM, not by arithmetic, so
// this path uses CUDA cores and reads K once:
//   logits kernel:  log2-domain logits x * log2(e)/sqrt(D) of every (logit row, key),
//                   stored per logit row with a row stride padded to 64 keys, and per
//                   CTA (max, sum of exp2) of every logit row over the multimodal keys of
//                   its tile.  Two variants:
//                   * rows8 (Hkv = 2 or 4, at most 8 rows per head group): a warp reads
//                     token rows coalesced, 16 lanes per KV head with 8 features each,
//                     holds its query slice in registers, and an 8-row reduce-scatter
//                     over the 16 lanes leaves one finished logit per lane pair;
//                   * general: one thread per key reads its whole token row and dots it
//                     with the group's query rows held in shared memory;
//   merge kernel:   per logit row, one block combines the CTA partials into lse2;
//   final kernel:   one thread per key sums exp2(logit - lse2) over all logit rows
//                   in a fixed order and scales by 1/(Hq n_q).
// The logits of the 10-minute 7B sequence with one query row take 15 MB and stay
// in L2 between the first and the last kernel.
#include <algorithm>
#include <cmath>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kThreads = 256;          // keys per CTA (general logits kernel, final kernel)
constexpr int kWarps = kThreads / 32;
constexpr int kRows8Tokens = 64;       // smallest key chunk of the rows8 logits kernel (sizes partials)
constexpr int kStrmWarps = 16;         // rows8 kernel: warps per CTA (lane 0 of the last also loads)
constexpr int kStrmThreads = kStrmWarps * 32;
constexpr int kStrmStages = 3;
constexpr int kStrmStageBytes = 65536; // K rows per stage: 64 tokens of 4 KV heads, 128 of 2
constexpr size_t kStrmSmem = static_cast<size_t>(kStrmStages) * kStrmStageBytes + 2 * kStrmStages * sizeof(uint64_t) +
                             kStrmWarps * 16 * sizeof(float2) + 16;
constexpr int kLogitPad = 64;          // logit row stride: the key count rounded up to this

struct NSeq {
  int32_t t0, len;
  int32_t q_off, n_q;
  int32_t unit_begin;                  // first 256-key CTA of this sequence (general logits, final)
  int32_t unit8_begin;                 // first chunk (CTA) of this sequence in the rows8 logits kernel
  int32_t nparts;                      // CTA partials of the logits kernel in use
  int32_t rows;                        // logit rows R = Hq * n_q
  int64_t lstride;                     // logit row stride: len rounded up to kLogitPad
  int64_t logit_base;                  // float offset of this sequence's logits [R][lstride]
  int64_t part_base;                   // float2 offset of its CTA partials [nparts][R]
  int64_t lse_base;                    // float offset of its lse2 [R]
};

struct NarrowPlan {
  int32_t nseq;
  int32_t total_units;
  int32_t total_units8;
  int32_t chunk;                       // keys per CTA of the rows8 kernel (a multiple of a stage)
  int32_t hq, hkv, group;
  float scale2;
  NSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int find_unit_seq(const NarrowPlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit_begin <= u) ++s;
  return s;
}

__device__ __forceinline__ int find_unit8_seq(const NarrowPlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit8_begin <= u) ++s;
  return s;
}

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
        // this warp's (max, sum of exp2) of the row over its multimodal keys
        const float wm = warp_max(mm ? y : -INFINITY);
        const float ws = warp_sum(mm && wm != -INFINITY ? ex2_approx(y - wm) : 0.f);
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

// rows8 logits kernel (Hkv = 2 or 4, at most 8 rows per head group): one CTA per chunk
// of a sequence's keys (about T / #SMs keys).  The chunk's K rows stream into a ring of
// kStrmStages shared-memory stages by bulk async copies (64 KB per stage: 64 tokens of
// 4 KV heads or 128 of 2); lane 0 of the last warp issues them and refills a slot once all
// warps have released it.  Warp w takes head pair w % NPAIR and the group of 8 keys
// (w / NPAIR) of every stage; lane l works on head 2 hp + (l >> 4) and features
// [8 (l & 15), 8 (l & 15) + 8), with its query slice in registers.  Per CTA it writes the
// (max, sum of exp2) of every logit row over its multimodal keys.
template <int NPAIR>
__global__ void __launch_bounds__(kStrmThreads, 1)
    score_narrow_rows8_kernel(const __grid_constant__ NarrowPlan plan, const uint16_t *__restrict__ q,
                              const uint8_t *__restrict__ k, int64_t k_stride, const uint8_t *__restrict__ modality,
                              float *__restrict__ logits, float2 *__restrict__ part, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t dsm[];
  uint8_t *stage_base = dsm;
  uint64_t *full = reinterpret_cast<uint64_t *>(dsm + kStrmStages * kStrmStageBytes);
  uint64_t *empty = full + kStrmStages;
  float2 *wst = reinterpret_cast<float2 *>(empty + kStrmStages);          // [warp][16]
  int *abort_flag = reinterpret_cast<int *>(wst + kStrmWarps * 16);
  const int c = blockIdx.x;
  const int s = find_unit8_seq(plan, c);
  const NSeq &sq = plan.seq[s];
  const int G = plan.group;
  const int rg = G * sq.n_q;
  if (rg == 0) return;                                   // no query row: nothing to score (CTA-uniform)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t row = static_cast<int64_t>(plan.hkv) * 256;
  const int stage_tok = kStrmStageBytes / static_cast<int>(row);
  const int tb = (c - sq.unit8_begin) * plan.chunk;
  const int te = min(sq.len, tb + plan.chunk);
  const int nst = (te - tb + stage_tok - 1) / stage_tok;
  const bool loader = warp == kStrmWarps - 1 && lane == 0;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStrmStages; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], kStrmWarps);
    }
    *abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int *abort_v = abort_flag;
  const uint8_t *kseq = k + static_cast<int64_t>(sq.t0) * k_stride;
  auto issue = [&](int n) {
    const int slot = n % kStrmStages;
    const int t = tb + n * stage_tok;
    const int cnt = min(stage_tok, te - t);
    uint8_t *dst = stage_base + static_cast<size_t>(slot) * kStrmStageBytes;
    mbar_arrive_expect_tx(&full[slot], static_cast<uint32_t>(cnt * row));
    if (k_stride == row) {
      bulk_load(dst, kseq + static_cast<int64_t>(t) * k_stride, static_cast<uint32_t>(cnt * row), &full[slot]);
    } else {
      for (int r = 0; r < cnt; ++r)
        bulk_load(dst + r * row, kseq + static_cast<int64_t>(t + r) * k_stride, static_cast<uint32_t>(row),
                  &full[slot]);
    }
  };
  int issued = 0;
  if (loader)
    for (; issued < kStrmStages && issued < nst; ++issued) issue(issued);

  const int hp = warp % NPAIR, grp = warp / NPAIR;
  const int h = 2 * hp + (lane >> 4), part16 = lane & 15;
  // query slice: rows j < rg of head group h (logit row (j / G) Hq + h G + j % G)
  float qf[8][8];
  const uint4 *qrow = reinterpret_cast<const uint4 *>(q + static_cast<int64_t>(sq.q_off) * plan.hq * 128);
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    uint4 w = make_uint4(0, 0, 0, 0);
    if (j < rg) w = __ldg(qrow + ((j / G) * plan.hq + h * G + j % G) * 16 + part16);
    bf16x8_to_f32(w, qf[j]);
  }
  const int r = (lane >> 1) & 7;                       // row this lane holds after the reduce-scatter
  const bool row_ok = r < rg;
  const int rho = row_ok ? (r / G) * plan.hq + h * G + r % G : 0;
  const bool b1 = lane & 8, b2 = lane & 4, b3 = lane & 2;
  float m = -INFINITY, ssum = 0.f;
  for (int n = 0; n < nst; ++n) {
    const int slot = n % kStrmStages;
    if (!__all_sync(0xffffffffu, mbar_wait(&full[slot], (n / kStrmStages) & 1u, kWaitLimitNs))) {
      if (lane == 0) {
        raise_device_error(err, APACK_ETIMEOUT, 71, c, n);
        *abort_v = 1;
      }
      break;
    }
    const int t0 = tb + n * stage_tok + grp * 8;
    const int valid = min(8, te - t0);
    if (valid > 0) {
      const uint8_t *ks = stage_base + static_cast<size_t>(slot) * kStrmStageBytes +
                          static_cast<size_t>(grp) * 8 * row + h * 256 + part16 * 16;
      const int tl = t0 + (lane & 7);
      const unsigned mmask = __ballot_sync(0xffffffffu, lane < 8 && tl < te && is_mm(modality[sq.t0 + tl]));
      float outv[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        float kf[8];
        bf16x8_to_f32(i < valid ? *reinterpret_cast<const uint4 *>(ks + i * row) : make_uint4(0, 0, 0, 0), kf);
        float acc[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          float2 a2 = make_float2(0.f, 0.f);
#pragma unroll
          for (int e = 0; e < 4; ++e)
            a2 = ffma2(make_float2(kf[2 * e], kf[2 * e + 1]), make_float2(qf[j][2 * e], qf[j][2 * e + 1]), a2);
          acc[j] = a2.x + a2.y;
        }
        // reduce-scatter over the 16 lanes of the head: lane bits 3, 2, 1 pick the row
        float v4[4], v2[2];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float send = b1 ? acc[e] : acc[e + 4];
          const float keep = b1 ? acc[e + 4] : acc[e];
          v4[e] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
        }
#pragma unroll
        for (int e = 0; e < 2; ++e) {
          const float send = b2 ? v4[e] : v4[e + 2];
          const float keep = b2 ? v4[e + 2] : v4[e];
          v2[e] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
        }
        float v1;
        {
          const float send = b3 ? v2[0] : v2[1];
          const float keep = b3 ? v2[1] : v2[0];
          v1 = keep + __shfl_xor_sync(0xffffffffu, send, 2);
        }
        v1 += __shfl_xor_sync(0xffffffffu, v1, 1);
        outv[i] = v1 * plan.scale2;
      }
      // running (max, sum of exp2) of this lane's row over the group's multimodal keys
      float cm = -INFINITY;
#pragma unroll
      for (int i = 0; i < 8; ++i)
        if ((mmask >> i) & 1u) cm = fmaxf(cm, outv[i]);
      if (cm != -INFINITY) {
        if (cm > m) {
          ssum *= ex2_approx(m - cm);
          m = cm;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if ((mmask >> i) & 1u) ssum += ex2_approx(outv[i] - m);
      }
      if (row_ok) {   // the lane pair writes the group's 8 logits of its row: 4 each
        const bool odd = lane & 1;
        const float4 w = odd ? make_float4(outv[4], outv[5], outv[6], outv[7])
                             : make_float4(outv[0], outv[1], outv[2], outv[3]);
        *reinterpret_cast<float4 *>(logits + sq.logit_base + static_cast<int64_t>(rho) * sq.lstride + t0 +
                                    (odd ? 4 : 0)) = w;
      }
    }
    __syncwarp();                        // this warp is done with the stage
    if (lane == 0) mbar_arrive(&empty[slot]);
    if (loader && issued < nst) {
      // every warp has released stage n: refill its slot
      if (!mbar_wait(&empty[slot], (n / kStrmStages) & 1u, kWaitLimitNs)) {
        raise_device_error(err, APACK_ETIMEOUT, 72, c, n);
        *abort_v = 1;
      } else {
        issue(issued);
        ++issued;
      }
    }
    __syncwarp();
    if (*abort_v) break;
  }
  // after an abort, stages may still be in flight: wait for them (bounded) before exit
  if (loader && *abort_v)
    for (int n = max(0, issued - kStrmStages); n < issued; ++n)
      mbar_wait(&full[n % kStrmStages], (n / kStrmStages) & 1u, kWaitLimitNs / 4);
  if ((lane & 1) == 0) wst[warp * 16 + (lane >> 1)] = make_float2(m, ssum);
  __syncthreads();
  if (*abort_v) return;
  // per (head, row): combine the warps of its head pair in key order
  if (threadIdx.x < 16 * NPAIR) {
    const int php = threadIdx.x >> 4, slot = threadIdx.x & 15;
    const int rr = slot & 7, hh = 2 * php + (slot >> 3);
    if (rr < rg) {
      float mx = -INFINITY;
      for (int g2 = 0; g2 < kStrmWarps / NPAIR; ++g2) mx = fmaxf(mx, wst[(g2 * NPAIR + php) * 16 + slot].x);
      float sum = 0.f;
      if (mx != -INFINITY)
        for (int g2 = 0; g2 < kStrmWarps / NPAIR; ++g2) {
          const float2 v = wst[(g2 * NPAIR + php) * 16 + slot];
          if (v.x != -INFINITY) sum += v.y * ex2_approx(v.x - mx);
        }
      const int rh = (rr / G) * plan.hq + hh * G + rr % G;
      part[sq.part_base + static_cast<int64_t>(c - sq.unit8_begin) * sq.rows + rh] = make_float2(mx, sum);
    }
  }
}

// One block per (sequence, logit row): lse2 over the CTA partials.  Each thread
// folds a fixed stride of partials, then a fixed-shape tree combines the
// threads: the order never depends on timing, so lse2 is deterministic.
__global__ void __launch_bounds__(kThreads)
    score_narrow_merge_kernel(const __grid_constant__ NarrowPlan plan, const float2 *__restrict__ part,
                              float *__restrict__ lse2) {
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
  float m = -INFINITY;
  for (int c = tid; c < ctas; c += kThreads) m = fmaxf(m, part[sq.part_base + static_cast<int64_t>(c) * sq.rows + rho].x);
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
  if (m != -INFINITY)
    for (int c = tid; c < ctas; c += kThreads) {
      const float2 v = part[sq.part_base + static_cast<int64_t>(c) * sq.rows + rho];
      if (v.x != -INFINITY) sum += v.y * exp2f(v.x - m);
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
  extern __shared__ __align__(16) float ls[];
  const int s = find_unit_seq(plan, blockIdx.x);
  const NSeq &sq = plan.seq[s];
  const int R = sq.rows;
  for (int i = threadIdx.x; i < R; i += kThreads) ls[i] = lse2[sq.lse_base + i];
  __syncthreads();
  const int kt = blockIdx.x - sq.unit_begin;
  const int key = sq.t0 + kt * kThreads + threadIdx.x;
  if (key >= sq.t0 + sq.len) return;
  float out = 0.f;
  if (sq.n_q > 0 && is_mm(modality[key])) {
    // eight independent sums, the loads of a block of 8 rows issued together
    const float *lp = logits + sq.logit_base + (key - sq.t0);
    float a[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
    for (int r0 = 0; r0 < R; r0 += 8) {
      float x[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        x[u] = r0 + u < R ? lp[static_cast<int64_t>(r0 + u) * sq.lstride] - ls[r0 + u] : -INFINITY;
#pragma unroll
      for (int u = 0; u < 8; ++u) a[u] += ex2_approx(x[u]);
    }
    out = (((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]))) / static_cast<float>(plan.hq * sq.n_q);
  }
  scores[key] = out;
}

template <int RG>
cudaError_t launch_logits(int grid, size_t smem, cudaStream_t stream, const NarrowPlan &P, const uint16_t *q,
                          const uint8_t *k, int64_t k_stride, const uint8_t *modality, float *logits, float2 *part) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(score_narrow_logits_kernel<RG>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize, 160 * 1024);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  score_narrow_logits_kernel<RG><<<grid, kThreads, smem, stream>>>(P, q, k, k_stride, modality, logits, part);
  return cudaGetLastError();
}

template <int NPAIR>
cudaError_t launch_rows8(int grid, cudaStream_t stream, const NarrowPlan &P, const uint16_t *q, const uint8_t *k,
                         int64_t k_stride, const uint8_t *modality, float *logits, float2 *part, DeviceError *err) {
  static bool attr = false;
  if (!attr) {
    const cudaError_t e = cudaFuncSetAttribute(score_narrow_rows8_kernel<NPAIR>,
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               static_cast<int>(kStrmSmem));
    if (e != cudaSuccess) return e;
    attr = true;
  }
  score_narrow_rows8_kernel<NPAIR><<<grid, kStrmThreads, kStrmSmem, stream>>>(P, q, k, k_stride, modality, logits,
                                                                             part, err);
  return cudaGetLastError();
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
    // rows8 kernel: K read by whole warps, query slice in registers
    int max_rg = 0;
    for (int i = 0; i < ns; ++i) {
      const int nq = seqs->cu_qlens_h[s0 + i + 1] - seqs->cu_qlens_h[s0 + i];
      max_rg = G * nq > max_rg ? G * nq : max_rg;
    }
    const bool rows8 = (hkv == 2 || hkv == 4) && max_rg <= 8;
    // rows8 chunk: about one CTA per SM over this launch's keys, a multiple of a stage
    int64_t launch_tokens = 0;
    for (int i = 0; i < ns; ++i) launch_tokens += seqs->cu_seqlens_h[s0 + i + 1] - seqs->cu_seqlens_h[s0 + i];
    const int64_t stage_tok = kStrmStageBytes / (static_cast<int64_t>(hkv) * 256);
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
      e = hkv == 4 ? launch_rows8<2>(units8, stream, P, q16, k8, k_token_stride, seqs->modality, logits, part, err)
                   : launch_rows8<1>(units8, stream, P, q16, k8, k_token_stride, seqs->modality, logits, part, err);
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
      score_narrow_merge_kernel<<<static_cast<unsigned>(rows_all), kThreads, 0, stream>>>(P, part, lse2);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    score_narrow_final_kernel<<<units, kThreads, static_cast<size_t>(max_rows) * sizeof(float), stream>>>(
        P, seqs->modality, logits, lse2, scores);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  return APACK_OK;
}

}  // namespace apack
