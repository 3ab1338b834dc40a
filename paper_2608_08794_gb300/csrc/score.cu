// score.cu -- relevance scores of Eq. inner_score (Sec. 3.2) on the tcgen05 tensor cores.
//
// I_i = 1/(Hq n_q) sum_h sum_r softmax_{j in S}(q_{r,h} . k_{j,g(h)} / sqrt(D))_i
//
// The softmax normaliser of every (query row, head) needs all keys of S before
// any per-key average can be formed, so the scores take two passes over K:
//
//  pass 1 (row statistics): D[row][key] = Q_tile . K_block^T with query rows in
//     TMEM lanes; each epilogue thread owns one row and keeps an online
//     (max, sum of exp2) over its keys.  Keys are split across CTAs; each
//     (split, row) writes a partial (max, sum) pair.
//  merge: per row, the partials combine into a log2-domain normaliser
//     lse2 = log2 sum_j 2^(x_j * log2(e)/sqrt(D)), stored per 256-row chunk.
//  pass 2 (column sums): D[key][row] = K_tile . Q_chunk^T with keys in TMEM
//     lanes; each thread owns one key and sums 2^(x*c - lse2[row]) over all
//     rows of all heads, then scales by 1/(Hq n_q).  Fixed order, no atomics.
//
// Both MMA passes: bf16 operands staged in 128-byte swizzled shared memory by
// TMA, fp32 accumulators in TMEM (two 256-column buffers so that the MMA of
// the next tile overlaps the exp2 epilogue of the current one), one TMA
// warp, one MMA-issuing warp and two epilogue warpgroups (each takes one half
// of the accumulator columns).  Persistent CTAs, one per SM.
#include <cmath>
#include <cstdio>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kThreads = 320;          // warp 0: TMA, warp 1: MMA, warps 2..9: epilogue
constexpr int kEpiThreads = 256;
constexpr uint32_t kTmemCols = 512;    // two accumulators of 256 fp32 columns
constexpr int kBlockKeys1 = 256;       // pass 1: keys per MMA (N)
constexpr int kTileKeys2 = 128;        // pass 2: keys per tile (M)
constexpr uint32_t kABytes = 128 * 256;        // 128 rows x 128 bf16
constexpr uint32_t kBBytes = 256 * 256;        // 256 rows x 128 bf16
constexpr uint32_t kAHalf = 128 * 128;         // offset of the second 64-element K half of A
constexpr uint32_t kBHalf = 256 * 128;         // ... of B
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 256);

struct SeqPlan {
  int32_t t0, len;        // token range of the sequence in the packed batch
  int32_t q_off, n_q;     // query rows in packed Q
  int32_t unit_begin;     // first work unit of this sequence in the launch
  int32_t n_qt;           // pass 1: query tiles of rows_tile1 tokens
  int32_t bps;            // pass 1: key blocks per split
  int32_t n_split;        // pass 1: splits
  int32_t chunk_base;     // index of this sequence's first lse2 chunk
  int32_t nch;            // pass 2: query chunks of rows_tile2 tokens per head
};

struct ScorePlan {
  int32_t nseq;
  int32_t total_units;
  int32_t hq, hkv, group;
  int32_t r1, r2;          // query tokens per tile in pass 1 / chunk in pass 2
  int32_t total_qrows;     // sum n_q over the whole batch
  float scale2;            // log2(e) / sqrt(D)
  SeqPlan seq[kSeqsPerLaunch];
};

struct __align__(8) Bars {
  uint64_t a_full[2], a_empty[2], b_full[2], b_empty[2], acc_full[2], acc_empty[2], drain;
  uint64_t comb_full, comb_empty;   // warpgroup 1 -> warpgroup 0 hand-off of per-row partials
  uint32_t tmem_base;
  volatile int32_t abort;
};

// Smem carve-up, identical for both passes: [A0][A1][B0][B1][Bars][combine].
constexpr uint32_t kOffA = 0;
constexpr uint32_t kOffB = 2 * kABytes;
constexpr uint32_t kOffBars = kOffB + 2 * kBBytes;
constexpr uint32_t kOffComb = kOffBars + 256;
constexpr uint32_t kSmemBytes = kOffComb + 128 * sizeof(float2) + 1024;   // + alignment slack

__device__ __forceinline__ int find_seq(const ScorePlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit_begin <= u) ++s;
  return s;
}

__device__ __forceinline__ bool is_mm(uint8_t m) { return m == APACK_MOD_AUDIO || m == APACK_MOD_VISUAL; }

// A wait that also gives up when another role has aborted.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Bars *bars, DeviceError *err,
                                              int where) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (bars->abort) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      bars->abort = 1;
      raise_device_error(err, APACK_ETIMEOUT, where);
      return false;
    }
  }
}

__device__ __forceinline__ uint8_t *aligned_smem(uint8_t *raw) {
  return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
}

__device__ void init_common(uint8_t *smem, Bars *bars, int warp, int lane) {
  // Zero both A and B buffers so that MMA rows no TMA box ever writes stay finite.
  for (uint32_t i = threadIdx.x; i < kOffBars / 16; i += blockDim.x)
    reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0, 0, 0, 0);
  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->a_full[i], 1);
      mbar_init(&bars->a_empty[i], 1);
      mbar_init(&bars->b_full[i], 1);
      mbar_init(&bars->b_empty[i], 1);
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], kEpiThreads / 32);
    }
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->comb_full, kEpiThreads / 2);
    mbar_init(&bars->comb_empty, kEpiThreads / 2);
    bars->abort = 0;
    fence_mbar_init();
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, kTmemCols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  (void)lane;
}

// Teardown: the MMA thread makes sure no MMA is in flight, then TMEM is freed.
__device__ void finish_common(Bars *bars, int warp, int lane, bool mma_thread, uint32_t drain_parity) {
  if (mma_thread && bars->abort) {
    tc_commit(&bars->drain);
    mbar_wait(&bars->drain, drain_parity, kWaitLimitNs / 4);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(bars->tmem_base, kTmemCols);
  (void)lane;
}

// Waits (bounded, ignoring the abort flag) for TMA loads that were issued
// but never consumed, so that no copy lands in shared memory after exit.
__device__ void drain_loads(uint64_t *full, const bool *pending, const uint32_t *parity, int n) {
  for (int i = 0; i < n; ++i)
    if (pending[i]) mbar_wait(&full[i], parity[i], kWaitLimitNs / 4);
}

// ------------------------------------------------------------------ pass 1
__device__ __forceinline__ void decode_unit1(const ScorePlan &p, int u, int &s, int &g, int &qt, int &b0, int &b1,
                                             int &split) {
  s = find_seq(p, u);
  const SeqPlan &sp = p.seq[s];
  const int local = u - sp.unit_begin;
  qt = local % sp.n_qt;
  const int pg = local / sp.n_qt;
  g = pg % p.hkv;
  split = pg / p.hkv;
  const int nb = (sp.len + kBlockKeys1 - 1) / kBlockKeys1;
  b0 = split * sp.bps;
  b1 = min(nb, b0 + sp.bps);
}

__global__ void __launch_bounds__(kThreads, 1)
    score_rowstats_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                          const __grid_constant__ ScorePlan plan, const uint8_t *__restrict__ modality,
                          float2 *__restrict__ part, DeviceError *err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = aligned_smem(smem_raw);
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  float2 *comb = reinterpret_cast<float2 *>(smem + kOffComb);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  init_common(smem, bars, warp, lane);
  const int G = plan.group;
  const uint32_t a_tx = 2u * G * plan.r1 * 128u;
  uint32_t drain_parity = 0;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[2] = {false, false};
      uint32_t pend_par[2] = {0, 0};
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        int s, g, qt, b0, b1, split;
        decode_unit1(plan, u, s, g, qt, b0, b1, split);
        const SeqPlan &sp = plan.seq[s];
        if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, err, 11)) { ok = false; break; }
        uint8_t *A = smem + kOffA + ai * kABytes;
        mbar_arrive_expect_tx(&bars->a_full[ai], a_tx);
        tma_load_3d(A, &qmap, &bars->a_full[ai], 0, g * G, sp.q_off + qt * plan.r1);
        tma_load_3d(A + kAHalf, &qmap, &bars->a_full[ai], 64, g * G, sp.q_off + qt * plan.r1);
        for (int b = b0; b < b1; ++b) {
          if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, err, 12)) { ok = false; break; }
          uint8_t *B = smem + kOffB + bi * kBBytes;
          mbar_arrive_expect_tx(&bars->b_full[bi], kBBytes);
          const int key0 = sp.t0 + b * kBlockKeys1;
          tma_load_3d(B, &kmap, &bars->b_full[bi], 0, g, key0);
          tma_load_3d(B + kBHalf, &kmap, &bars->b_full[bi], 64, g, key0);
          pend[bi] = true;
          pend_par[bi] = bph;
          if (++bi == 2) { bi = 0; bph ^= 1; }
        }
        if (++ai == 2) { ai = 0; aph ^= 1; }
      }
      if (!ok) drain_loads(bars->b_full, pend, pend_par, 2);
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        int s, g, qt, b0, b1, split;
        decode_unit1(plan, u, s, g, qt, b0, b1, split);
        if (!wait_or_abort(&bars->a_full[ai], aph, bars, err, 13)) { ok = false; break; }
        const uint32_t a_base = smem_u32(smem + kOffA + ai * kABytes);
        for (int b = b0; b < b1; ++b) {
          if (!wait_or_abort(&bars->b_full[bi], bph, bars, err, 14)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, err, 15)) { ok = false; break; }
          tc_fence_after();
          const uint32_t b_base = smem_u32(smem + kOffB + bi * kBBytes);
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t ao = (kk >> 2) * kAHalf + (kk & 3) * 32;
            const uint32_t bo = (kk >> 2) * kBHalf + (kk & 3) * 32;
            tc_mma_bf16(tmem + ci * 256, smem_desc_sw128(a_base + ao), smem_desc_sw128(b_base + bo), kIdesc,
                        kk > 0 ? 1u : 0u);
          }
          tc_commit(&bars->b_empty[bi]);
          tc_commit(&bars->acc_full[ci]);
          if (++bi == 2) { bi = 0; bph ^= 1; }
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
        if (!ok) break;
        tc_commit(&bars->a_empty[ai]);
        if (++ai == 2) { ai = 0; aph ^= 1; }
      }
    }
  } else {
    // Epilogue: warp w reads TMEM lanes 32*(w%4).., column half wg.
    const int wg = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int row = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const float c2 = plan.scale2;
    int ci = 0;
    uint32_t cph = 0, xph = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
      int s, g, qt, b0, b1, split;
      decode_unit1(plan, u, s, g, qt, b0, b1, split);
      const SeqPlan &sp = plan.seq[s];
      const int t_end = sp.t0 + sp.len;
      float m = -INFINITY, sum = 0.f;
      for (int b = b0; b < b1; ++b) {
        if (!wait_or_abort(&bars->acc_full[ci], cph, bars, err, 16)) { ok = false; break; }
        tc_fence_after();
        const int key_base = sp.t0 + b * kBlockKeys1 + wg * 128;
        const uint32_t tcol = bars->tmem_base + lane_off + ci * 256 + wg * 128;
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
          float v[32];
          tmem_ld32(tcol + c * 32, v);
          const int key = key_base + c * 32 + lane;
          const bool valid = key < t_end && is_mm(modality[key]);
          const uint32_t mask = __ballot_sync(0xffffffffu, valid);
          tmem_ld_wait();
          if (mask == 0u) continue;
          float mx = -INFINITY;
          if (mask == 0xffffffffu) {
#pragma unroll
            for (int i = 0; i < 32; ++i) mx = fmaxf(mx, v[i]);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if ((mask >> i) & 1u) mx = fmaxf(mx, v[i]);
          }
          mx *= c2;
          if (mx > m) {
            sum *= ex2_approx(m - mx);
            m = mx;
          }
          float t0 = 0.f, t1 = 0.f;
          if (mask == 0xffffffffu) {
#pragma unroll
            for (int i = 0; i < 32; i += 2) {
              t0 += ex2_approx(fmaf(v[i], c2, -m));
              t1 += ex2_approx(fmaf(v[i + 1], c2, -m));
            }
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
              if ((mask >> i) & 1u) t0 += ex2_approx(fmaf(v[i], c2, -m));
          }
          sum += t0 + t1;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->acc_empty[ci]);
        if (++ci == 2) { ci = 0; cph ^= 1; }
      }
      if (!ok) break;
      // Combine the two column halves of the row, then store the partial.
      if (wg == 1) {
        if (!wait_or_abort(&bars->comb_empty, xph ^ 1, bars, err, 17)) break;
        comb[row] = make_float2(m, sum);
        mbar_arrive(&bars->comb_full);
      } else {
        if (!wait_or_abort(&bars->comb_full, xph, bars, err, 18)) break;
        const float2 o = comb[row];
        mbar_arrive(&bars->comb_empty);
        const float mm = fmaxf(m, o.x);
        float tot = 0.f;
        if (mm != -INFINITY) tot = sum * ex2_approx(m - mm) + o.y * ex2_approx(o.x - mm);
        const int rloc = row / G, j = row - rloc * G;
        const int r = qt * plan.r1 + rloc;
        if (row < G * plan.r1 && r < sp.n_q) {
          const int qrow = sp.q_off + r;
          part[(static_cast<size_t>(split) * plan.total_qrows + qrow) * plan.hq + g * G + j] = make_float2(mm, tot);
        }
      }
      xph ^= 1;
    }
  }
  finish_common(bars, warp, lane, warp == 1 && lane == 0, drain_parity);
}

// ------------------------------------------------------------------ merge
// One thread per lse2 entry: (sequence, KV head, chunk, column).
__global__ void lse_merge_kernel(const __grid_constant__ ScorePlan plan, const float2 *__restrict__ part,
                                 float *__restrict__ lse2, int64_t n_entries, int64_t entry_base) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n_entries) return;
  const int64_t chunk = entry_base / 256 + e / 256;
  const int col = static_cast<int>(e % 256);
  int s = 0;
  while (s + 1 < plan.nseq && plan.seq[s + 1].chunk_base <= chunk) ++s;
  const SeqPlan &sp = plan.seq[s];
  const int local = static_cast<int>(chunk - sp.chunk_base);
  const int g = local / sp.nch, c = local - g * sp.nch;
  const int G = plan.group;
  const int rloc = col / G, j = col - rloc * G;
  const int r = c * plan.r2 + rloc;
  float out = INFINITY;   // padding columns contribute exp2(-inf) = 0 in pass 2
  if (col < G * plan.r2 && r < sp.n_q) {
    const int qrow = sp.q_off + r;
    const int h = g * G + j;
    float mm = -INFINITY;
    for (int p = 0; p < sp.n_split; ++p)
      mm = fmaxf(mm, part[(static_cast<size_t>(p) * plan.total_qrows + qrow) * plan.hq + h].x);
    if (mm == -INFINITY) {
      out = -INFINITY;
    } else {
      float tot = 0.f;
      for (int p = 0; p < sp.n_split; ++p) {
        const float2 v = part[(static_cast<size_t>(p) * plan.total_qrows + qrow) * plan.hq + h];
        tot += v.y * exp2f(v.x - mm);
      }
      out = mm + log2f(tot);
    }
  }
  lse2[chunk * 256 + col] = out;
}

// ------------------------------------------------------------------ pass 2
__device__ __forceinline__ void decode_unit2(const ScorePlan &p, int u, int &s, int &kt) {
  s = find_seq(p, u);
  kt = u - p.seq[s].unit_begin;
}

__global__ void __launch_bounds__(kThreads, 1)
    score_colsum_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                        const __grid_constant__ ScorePlan plan, const uint8_t *__restrict__ modality,
                        const float *__restrict__ lse2, float *__restrict__ scores, DeviceError *err) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t *smem = aligned_smem(smem_raw);
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  float *comb = reinterpret_cast<float *>(smem + kOffComb);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  init_common(smem, bars, warp, lane);
  const int G = plan.group;
  const uint32_t b_tx = 2u * G * plan.r2 * 128u;
  uint32_t drain_parity = 0;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[2] = {false, false}, apend[2] = {false, false};
      uint32_t pend_par[2] = {0, 0}, apend_par[2] = {0, 0};
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        int s, kt;
        decode_unit2(plan, u, s, kt);
        const SeqPlan &sp = plan.seq[s];
        if (sp.nch == 0) continue;
        const int key0 = sp.t0 + kt * kTileKeys2;
        for (int g = 0; ok && g < plan.hkv; ++g) {
          if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, err, 21)) { ok = false; break; }
          uint8_t *A = smem + kOffA + ai * kABytes;
          mbar_arrive_expect_tx(&bars->a_full[ai], kABytes);
          tma_load_3d(A, &kmap, &bars->a_full[ai], 0, g, key0);
          tma_load_3d(A + kAHalf, &kmap, &bars->a_full[ai], 64, g, key0);
          apend[ai] = true;
          apend_par[ai] = aph;
          for (int c = 0; c < sp.nch; ++c) {
            if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, err, 22)) { ok = false; break; }
            uint8_t *B = smem + kOffB + bi * kBBytes;
            mbar_arrive_expect_tx(&bars->b_full[bi], b_tx);
            const int qrow0 = sp.q_off + c * plan.r2;
            tma_load_3d(B, &qmap, &bars->b_full[bi], 0, g * G, qrow0);
            tma_load_3d(B + kBHalf, &qmap, &bars->b_full[bi], 64, g * G, qrow0);
            pend[bi] = true;
            pend_par[bi] = bph;
            if (++bi == 2) { bi = 0; bph ^= 1; }
          }
          if (++ai == 2) { ai = 0; aph ^= 1; }
        }
      }
      if (!ok) {
        drain_loads(bars->b_full, pend, pend_par, 2);
        drain_loads(bars->a_full, apend, apend_par, 2);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        int s, kt;
        decode_unit2(plan, u, s, kt);
        const SeqPlan &sp = plan.seq[s];
        if (sp.nch == 0) continue;
        for (int g = 0; ok && g < plan.hkv; ++g) {
          if (!wait_or_abort(&bars->a_full[ai], aph, bars, err, 23)) { ok = false; break; }
          const uint32_t a_base = smem_u32(smem + kOffA + ai * kABytes);
          for (int c = 0; c < sp.nch; ++c) {
            if (!wait_or_abort(&bars->b_full[bi], bph, bars, err, 24)) { ok = false; break; }
            if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, err, 25)) { ok = false; break; }
            tc_fence_after();
            const uint32_t b_base = smem_u32(smem + kOffB + bi * kBBytes);
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
              const uint32_t ao = (kk >> 2) * kAHalf + (kk & 3) * 32;
              const uint32_t bo = (kk >> 2) * kBHalf + (kk & 3) * 32;
              tc_mma_bf16(tmem + ci * 256, smem_desc_sw128(a_base + ao), smem_desc_sw128(b_base + bo), kIdesc,
                          kk > 0 ? 1u : 0u);
            }
            tc_commit(&bars->b_empty[bi]);
            tc_commit(&bars->acc_full[ci]);
            if (++bi == 2) { bi = 0; bph ^= 1; }
            if (++ci == 2) { ci = 0; cph ^= 1; }
          }
          if (!ok) break;
          tc_commit(&bars->a_empty[ai]);
          if (++ai == 2) { ai = 0; aph ^= 1; }
        }
      }
    }
  } else {
    const int wg = (warp - 2) >> 2;
    const int quad = warp & 3;
    const int klane = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const float c2 = plan.scale2;
    int ci = 0;
    uint32_t cph = 0, xph = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
      int s, kt;
      decode_unit2(plan, u, s, kt);
      const SeqPlan &sp = plan.seq[s];
      float acc = 0.f;
      for (int g = 0; ok && g < plan.hkv && sp.nch > 0; ++g) {
        for (int c = 0; c < sp.nch; ++c) {
          if (!wait_or_abort(&bars->acc_full[ci], cph, bars, err, 26)) { ok = false; break; }
          tc_fence_after();
          const float4 *lp = reinterpret_cast<const float4 *>(
              lse2 + (static_cast<int64_t>(sp.chunk_base) + g * sp.nch + c) * 256 + wg * 128);
          const uint32_t tcol = bars->tmem_base + lane_off + ci * 256 + wg * 128;
#pragma unroll 1
          for (int cc = 0; cc < 4; ++cc) {
            float v[32];
            tmem_ld32(tcol + cc * 32, v);
            tmem_ld_wait();
            float a0 = 0.f, a1 = 0.f;
#pragma unroll
            for (int i = 0; i < 32; i += 4) {
              const float4 L = __ldg(lp + cc * 8 + i / 4);
              a0 += ex2_approx(fmaf(v[i], c2, -L.x));
              a1 += ex2_approx(fmaf(v[i + 1], c2, -L.y));
              a0 += ex2_approx(fmaf(v[i + 2], c2, -L.z));
              a1 += ex2_approx(fmaf(v[i + 3], c2, -L.w));
            }
            acc += a0 + a1;
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[ci]);
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
      }
      if (!ok) break;
      if (wg == 1) {
        if (!wait_or_abort(&bars->comb_empty, xph ^ 1, bars, err, 27)) break;
        comb[klane] = acc;
        mbar_arrive(&bars->comb_full);
      } else {
        if (!wait_or_abort(&bars->comb_full, xph, bars, err, 28)) break;
        const float other = comb[klane];
        mbar_arrive(&bars->comb_empty);
        const int key = sp.t0 + kt * kTileKeys2 + klane;
        if (key < sp.t0 + sp.len) {
          float out = 0.f;
          if (is_mm(modality[key]) && sp.n_q > 0)
            out = (acc + other) / static_cast<float>(plan.hq * sp.n_q);
          scores[key] = out;
        }
      }
      xph ^= 1;
    }
  }
  finish_common(bars, warp, lane, warp == 1 && lane == 0, drain_parity);
}

// ------------------------------------------------------------------ host side
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  if (!fn) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 3-D bf16 map: dims {128, mid, rows}, byte strides {mid_stride, row_stride}, box {64, box_mid, box_rows}.
bool make_map(CUtensorMap *map, const void *base, uint64_t mid, uint64_t rows, uint64_t mid_stride,
              uint64_t row_stride, uint32_t box_mid, uint32_t box_rows) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t dims[3] = {128, mid, rows};
  cuuint64_t strides[2] = {mid_stride, row_stride};
  cuuint32_t box[3] = {64, box_mid, box_rows};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool g_attr_done = false;

}  // namespace

apack_status run_score(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                       float *scores, void *ws, cudaStream_t stream) {
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (!q || !k || !scores || !ws) return APACK_EINVAL;
  if ((reinterpret_cast<uintptr_t>(q) & 15) || (reinterpret_cast<uintptr_t>(k) & 15) || (k_token_stride & 15) ||
      k_token_stride < static_cast<int64_t>(seqs->num_kv_heads) * 256)
    return APACK_EINVAL;
  const int B = seqs->num_seqs;
  const int hq = seqs->num_q_heads, hkv = seqs->num_kv_heads, G = hq / hkv;
  if (G > 128 || hkv > 256) return APACK_EUNSUPPORTED;
  if (T == 0) return APACK_OK;
  const WsLayout L = workspace_layout(seqs);
  uint8_t *wsb = static_cast<uint8_t *>(ws);
  DeviceError *err = reinterpret_cast<DeviceError *>(wsb + L.err_off);
  float2 *part = reinterpret_cast<float2 *>(wsb + L.part_off);
  float *lse2 = reinterpret_cast<float *>(wsb + L.lse_off);

  if (!g_attr_done) {
    if (check_cuda(cudaFuncSetAttribute(score_rowstats_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        kSmemBytes)) != APACK_OK ||
        check_cuda(cudaFuncSetAttribute(score_colsum_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                        kSmemBytes)) != APACK_OK)
      return APACK_ECUDA;
    g_attr_done = true;
  }
  const int r1 = rows_tile1(G), r2 = rows_tile2(G);
  CUtensorMap qmap1, kmap1, qmap2, kmap2;
  const uint64_t nq_rows = static_cast<uint64_t>(NQ > 0 ? NQ : 1);
  if (!make_map(&qmap1, q, hq, nq_rows, 256, static_cast<uint64_t>(hq) * 256, G, r1) ||
      !make_map(&kmap1, k, hkv, T, 256, k_token_stride, 1, kBlockKeys1) ||
      !make_map(&qmap2, q, hq, nq_rows, 256, static_cast<uint64_t>(hq) * 256, G, r2) ||
      !make_map(&kmap2, k, hkv, T, 256, k_token_stride, 1, kTileKeys2))
    return APACK_ECUDA;

  const int sms = device_sm_count();
  int64_t chunk_base = 0;
  for (int s0 = 0; s0 < B; s0 += kSeqsPerLaunch) {
    const int ns = (B - s0 < kSeqsPerLaunch) ? (B - s0) : kSeqsPerLaunch;
    ScorePlan P{};
    P.nseq = ns;
    P.hq = hq;
    P.hkv = hkv;
    P.group = G;
    P.r1 = r1;
    P.r2 = r2;
    P.total_qrows = static_cast<int32_t>(NQ);
    P.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(APACK_HEAD_DIM)));
    // Pass 1 work: key blocks x query tiles x heads, split so that the units
    // number a few per SM.
    int64_t work = 0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      const int len = seqs->cu_seqlens_h[b + 1] - seqs->cu_seqlens_h[b];
      const int nq = seqs->cu_qlens_h[b + 1] - seqs->cu_qlens_h[b];
      const int64_t nb = (len + kBlockKeys1 - 1) / kBlockKeys1;
      work += nb * hkv * ((nq + r1 - 1) / r1);
    }
    const int64_t target_units = 4LL * sms;
    int64_t bps_all = (work + target_units - 1) / (target_units > 0 ? target_units : 1);
    if (bps_all < 2) bps_all = 2;
    int units1 = 0, units2 = 0;
    int64_t chunks = 0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      SeqPlan &sp = P.seq[i];
      sp.t0 = seqs->cu_seqlens_h[b];
      sp.len = seqs->cu_seqlens_h[b + 1] - sp.t0;
      sp.q_off = seqs->cu_qlens_h[b];
      sp.n_q = seqs->cu_qlens_h[b + 1] - sp.q_off;
      const int nb = (sp.len + kBlockKeys1 - 1) / kBlockKeys1;
      sp.n_qt = (sp.n_q + r1 - 1) / r1;
      int bps = static_cast<int>(bps_all);
      if ((nb + bps - 1) / bps > kMaxSplits) bps = (nb + kMaxSplits - 1) / kMaxSplits;
      sp.bps = bps > 0 ? bps : 1;
      sp.n_split = (sp.n_q > 0 && nb > 0) ? (nb + sp.bps - 1) / sp.bps : 0;
      sp.unit_begin = units1;
      units1 += sp.n_split * hkv * sp.n_qt;
      sp.nch = (sp.n_q + r2 - 1) / r2;
      sp.chunk_base = static_cast<int32_t>(chunk_base + chunks);
      chunks += static_cast<int64_t>(hkv) * sp.nch;
    }
    // Pass 1.
    P.total_units = units1;
    if (units1 > 0) {
      const int grid = units1 < sms ? units1 : sms;
      score_rowstats_kernel<<<grid, kThreads, kSmemBytes, stream>>>(qmap1, kmap1, P, seqs->modality, part, err);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    // Merge into the per-chunk log2 normalisers.
    if (chunks > 0) {
      const int64_t n_entries = chunks * 256;
      const int threads = 256;
      const int64_t blocks = (n_entries + threads - 1) / threads;
      lse_merge_kernel<<<static_cast<unsigned>(blocks), threads, 0, stream>>>(P, part, lse2, n_entries,
                                                                              chunk_base * 256);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    // Pass 2: one unit per 128-key tile of each sequence.
    for (int i = 0; i < ns; ++i) {
      P.seq[i].unit_begin = units2;
      units2 += (P.seq[i].len + kTileKeys2 - 1) / kTileKeys2;
    }
    P.total_units = units2;
    if (units2 > 0) {
      const int grid = units2 < sms ? units2 : sms;
      score_colsum_kernel<<<grid, kThreads, kSmemBytes, stream>>>(qmap2, kmap2, P, seqs->modality, lse2, scores,
                                                                  err);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    chunk_base += chunks;
  }
  return APACK_OK;
}

}  // namespace apack
