// score_narrow_tc.cu -- logits of the narrow scoring path (few query rows per KV head group,
// e.g. the paper's last query token: Sec. 3.2, Eq. inner_score; Table S-hparams) on the
// tcgen05 tensor cores.
//
// One CTA per chunk of a sequence's keys (about T / #SMs keys).  For every 128-key tile and KV
// head h, the MMA computes D[key][row] = K_h[key] . Q_h[row] with keys as M = 128 and the
// head group's query rows as N = 16 (zero rows pad the group's <= 8 rows): bf16 operands in
// 128-byte-swizzled shared memory, fp32 accumulators in TMEM.
//   warp 0, one lane:  TMA loads of the K tiles (one stage = one head of one tile, 32 KB)
//   warp 1, one lane:  TMEM allocation and the MMAs (8 per stage), commits to mbarriers
//   warps 2..:         epilogue, one warpgroup per KV head, one key per thread: reads its
//                      head's 16 TMEM columns of the tile,
//                      stores the log2-domain logits (row-major per logit row, as the
//                      CUDA-core path) and keeps, per (head, row), the running (max, sum of
//                      exp2) over its multimodal keys.
// At the end the CTA merges the 128 per-thread states per logit row in thread order and
// writes one (max, sum) partial per row: the merge and final kernels of the narrow path
// consume the logits and partials unchanged.  Every wait is bounded.
#include <cmath>

#include "internal.cuh"
#include "narrow_plan.cuh"
#include "ptx.cuh"

namespace apack {
namespace {

constexpr int kTcM = 128;                          // keys per tile (MMA M)
constexpr int kTcN = 16;                           // query rows per head group, padded (MMA N)
constexpr int kTcRows = 8;                         // query rows per head group supported
constexpr int kTcStages = 6;                       // K ring: one (tile, head) per stage
constexpr int kTcHalf = kTcM * 128;                // 64 dims x 128 keys x 2 B = 16 KB
constexpr int kTcStageBytes = 2 * kTcHalf;         // 32 KB
constexpr int kTcQHalf = kTcN * 128;               // 2 KB: 64 dims of the 16 rows
// epilogue: one warpgroup (4 warps, one per TMEM lane quadrant) per KV head
template <int HKV>
__host__ __device__ constexpr int tc_epi_warps() { return 4 * HKV; }
template <int HKV>
__host__ __device__ constexpr int tc_threads() { return 64 + 32 * tc_epi_warps<HKV>(); }   // warp 0 TMA, warp 1 MMA, epilogue
constexpr uint32_t kTcIdesc = idesc_bf16_f32(kTcM, kTcN);

struct __align__(8) TcBars {
  uint64_t k_full[kTcStages], k_empty[kTcStages], acc_full[2], acc_empty[2], drain;
  uint32_t tmem_base;
  volatile int32_t abort;
};

template <int HKV>
struct TcLayout {
  static constexpr uint32_t kOffQ = kTcStages * kTcStageBytes;           // 1024-aligned
  static constexpr uint32_t kOffBars = kOffQ + HKV * 2 * kTcQHalf;
  static constexpr uint32_t kBytes = kOffBars + 256;
  static constexpr uint32_t kTmemCols = 2 * HKV * kTcN < 32 ? 32 : 2 * HKV * kTcN;   // power of 2 here
};

__device__ __forceinline__ bool tc_wait(uint64_t *bar, uint32_t parity, TcBars *bars, DeviceError *err, int where) {
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

__device__ __forceinline__ bool is_mm_tc(uint8_t m) { return m == APACK_MOD_AUDIO || m == APACK_MOD_VISUAL; }

template <int HKV>
__global__ void __launch_bounds__(tc_threads<HKV>(), 1)
    score_narrow_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ NarrowPlan plan,
                           const uint16_t *__restrict__ q, const uint8_t *__restrict__ modality,
                           float *__restrict__ logits, float2 *__restrict__ part, DeviceError *err) {
  pdl_wait_and_release();
  using Lay = TcLayout<HKV>;
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 80);
    return;
  }
  uint8_t *ring = smem;
  uint8_t *qs = smem + Lay::kOffQ;
  TcBars *bars = reinterpret_cast<TcBars *>(smem + Lay::kOffBars);
  const int c = blockIdx.x;
  const int s = find_unit8_seq(plan, c);
  const NSeq &sq = plan.seq[s];
  const int G = plan.group;
  const int rg = G * sq.n_q;
  if (rg == 0) return;                                 // no query row: nothing to score (CTA-uniform)
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int tb = (c - sq.unit8_begin) * plan.chunk;
  const int te = min(sq.len, tb + plan.chunk);
  const int ntiles = (te - tb + kTcM - 1) / kTcM;

  // query tiles in the 128-byte-swizzled K-major layout: row r, 16-byte chunk cc of a 64-dim
  // half sits at chunk cc ^ (r & 7) of the row's 128 bytes (every ring stage the MMAs read is
  // written whole by its TMA load, rows past the cache as zeros)
  for (int idx = threadIdx.x; idx < HKV * kTcN * 16; idx += tc_threads<HKV>()) {
    const int h = idx / (kTcN * 16), rem = idx % (kTcN * 16);
    const int row = rem / 16, ch = rem % 16;
    const int half = ch >> 3, cc = ch & 7;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (row < rg) {
      const int rho = (row / G) * plan.hq + h * G + row % G;
      v = __ldg(reinterpret_cast<const uint4 *>(q + (static_cast<int64_t>(sq.q_off) * plan.hq + rho) * 128) + ch);
    }
    *reinterpret_cast<uint4 *>(qs + h * 2 * kTcQHalf + half * kTcQHalf + (row >> 3) * 1024 + (row & 7) * 128 +
                               ((cc ^ (row & 7)) << 4)) = v;
  }
  if (threadIdx.x == 0) {
    for (int i = 0; i < kTcStages; ++i) {
      mbar_init(&bars->k_full[i], 1);
      mbar_init(&bars->k_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], tc_epi_warps<HKV>());
    }
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  fence_proxy_async_smem();   // generic-proxy writes of the tiles -> visible to TMA and the MMA
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, Lay::kTmemCols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  const int nstage = ntiles * HKV;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&kmap);
      int n = 0;
      bool pend[kTcStages] = {};
      uint32_t pend_par[kTcStages] = {};
      for (; n < nstage; ++n) {
        const int slot = n % kTcStages;
        if (n >= kTcStages && !tc_wait(&bars->k_empty[slot], ((n / kTcStages) - 1) & 1u, bars, err, 81)) break;
        const int t = n / HKV, h = n % HKV;
        uint8_t *dst = ring + slot * kTcStageBytes;
        mbar_arrive_expect_tx(&bars->k_full[slot], kTcStageBytes);
        const int key0 = sq.t0 + tb + t * kTcM;
        tma_load_3d(dst, &kmap, &bars->k_full[slot], 0, h, key0);
        tma_load_3d(dst + kTcHalf, &kmap, &bars->k_full[slot], 64, h, key0);
        pend[slot] = true;
        pend_par[slot] = (n / kTcStages) & 1u;
      }
      if (bars->abort)   // loads issued but not consumed: let them land before the CTA exits
        for (int i = 0; i < kTcStages; ++i)
          if (pend[i]) mbar_wait(&bars->k_full[i], pend_par[i], kWaitLimitNs / 4);
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      const uint32_t tmem = bars->tmem_base;
      const uint32_t q_base = smem_u32(qs);
      bool ok = true;
      for (int t = 0; ok && t < ntiles; ++t) {
        const int buf = t & 1;
        if (t >= 2 && !tc_wait(&bars->acc_empty[buf], ((t >> 1) - 1) & 1u, bars, err, 82)) break;
        for (int h = 0; h < HKV; ++h) {
          const int n = t * HKV + h, slot = n % kTcStages;
          if (!tc_wait(&bars->k_full[slot], (n / kTcStages) & 1u, bars, err, 83)) { ok = false; break; }
          tc_fence_after();
          const uint32_t a_base = smem_u32(ring + slot * kTcStageBytes);
          const uint32_t b_base = q_base + h * 2 * kTcQHalf;
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) {
            const uint32_t ao = (kk >> 2) * kTcHalf + (kk & 3) * 32;
            const uint32_t bo = (kk >> 2) * kTcQHalf + (kk & 3) * 32;
            tc_mma_bf16(tmem + buf * HKV * kTcN + h * kTcN, smem_desc_sw128(a_base + ao), smem_desc_sw128(b_base + bo),
                        kTcIdesc, kk > 0 ? 1u : 0u);
          }
          tc_commit(&bars->k_empty[slot]);
        }
        if (ok) tc_commit(&bars->acc_full[buf]);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    constexpr int HH = 1;                             // heads per epilogue warpgroup
    const int ew = warp - 2;
    const int quad = warp & 3;                        // TMEM lanes 32 * (warp % 4) ..
    const int hg = ew >> 2;                           // heads hg * HH ..
    const int kt = quad * 32 + lane;                  // key within the tile
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    float m[HH][kTcRows], sum[HH][kTcRows];
#pragma unroll
    for (int h = 0; h < HH; ++h)
#pragma unroll
      for (int j = 0; j < kTcRows; ++j) {
        m[h][j] = -INFINITY;
        sum[h][j] = 0.f;
      }
    const float c2 = plan.scale2;
    // modality of this thread's key, one tile ahead
    uint8_t mod_next = (tb + kt < te) ? modality[sq.t0 + tb + kt] : 0;
    for (int t = 0; t < ntiles; ++t) {
      const int buf = t & 1;
      const int key = tb + t * kTcM + kt;
      const bool valid = key < te;
      const bool mm = valid && is_mm_tc(mod_next);
      if (t + 1 < ntiles) mod_next = (key + kTcM < te) ? modality[sq.t0 + key + kTcM] : 0;
      // warp-uniform: tcgen05.ld below is a warp-collective instruction
      if (!__all_sync(0xffffffffu, tc_wait(&bars->acc_full[buf], (t >> 1) & 1u, bars, err, 84))) break;
      tc_fence_after();
      uint32_t r[HH * kTcN];
      const uint32_t taddr = bars->tmem_base + lane_off + buf * HKV * kTcN + hg * HH * kTcN;
      tmem_ld16(taddr, r);
      tmem_wait16(r);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->acc_empty[buf]);   // the values are in registers
#pragma unroll
      for (int hh = 0; hh < HH; ++hh)
#pragma unroll
        for (int j = 0; j < kTcRows; ++j) {
          if (j >= rg) continue;
          const int h = hg * HH + hh;
          const float y = __uint_as_float(r[hh * kTcN + j]) * c2;
          const int rho = (j / G) * plan.hq + h * G + j % G;
          if (valid) logits[sq.logit_base + static_cast<int64_t>(rho) * sq.lstride + key] = y;
          // the row's denominator: multimodal keys, or (causal rows) every key up to its position
          if (plan.causal ? (valid && key <= sq.q_pos + j / G) : mm) {
            const float mn = fmaxf(m[hh][j], y);
            sum[hh][j] = sum[hh][j] * ex2_approx(m[hh][j] - mn) + ex2_approx(y - mn);
            m[hh][j] = mn;
          }
        }
    }
    // per-thread states into the (drained) ring after everyone is done, below
    tc_fence_before();
    __syncthreads();
    if (!bars->abort) {
      float2 *red = reinterpret_cast<float2 *>(ring);   // [128 keys][HKV * 8]
#pragma unroll
      for (int hh = 0; hh < HH; ++hh)
#pragma unroll
        for (int j = 0; j < kTcRows; ++j)
          red[kt * (HKV * kTcRows) + (hg * HH + hh) * kTcRows + j] = make_float2(m[hh][j], sum[hh][j]);
    }
    asm volatile("bar.sync 1, %0;" ::"n"(tc_epi_warps<HKV>() * 32) : "memory");
    if (!bars->abort) {
      // one warp per (head, row): each lane folds 4 of the 128 per-key states, then a fixed
      // shuffle tree combines the lanes (deterministic order)
      const float2 *red = reinterpret_cast<const float2 *>(ring);
      for (int e = ew; e < HKV * kTcRows; e += tc_epi_warps<HKV>()) {
        const int h = e / kTcRows, j = e % kTcRows;
        if (j >= rg) continue;                          // uniform over the warp
        float2 v[kTcM / 32];
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < kTcM / 32; ++i) {
          v[i] = red[(lane + 32 * i) * (HKV * kTcRows) + e];
          mx = fmaxf(mx, v[i].x);
        }
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
        float tot = 0.f;
        if (mx != -INFINITY)
#pragma unroll
          for (int i = 0; i < kTcM / 32; ++i)
            if (v[i].x != -INFINITY) tot += v[i].y * ex2_approx(v[i].x - mx);
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, off);
        if (lane == 0) {
          const int rho = (j / G) * plan.hq + h * G + j % G;
          part[sq.part_base + static_cast<int64_t>(c - sq.unit8_begin) * sq.rows + rho] = make_float2(mx, tot);
        }
      }
    }
    // teardown below
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(bars->tmem_base, Lay::kTmemCols);
    return;
  }
  // producer and MMA warps: after an abort make sure no MMA is in flight, then meet the
  // epilogue at its two CTA barriers and free TMEM
  if (warp == 1 && lane == 0 && bars->abort) {
    tc_commit(&bars->drain);
    mbar_wait(&bars->drain, 0, kWaitLimitNs / 4);
  }
  tc_fence_before();
  __syncthreads();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(bars->tmem_base, Lay::kTmemCols);
}

}  // namespace

// Launches the tensor-core logits kernel for Hkv = 2 or 4 and at most 8 rows per head group.
cudaError_t launch_narrow_tc(int grid, cudaStream_t stream, const CUtensorMap &kmap, const NarrowPlan &P,
                             const uint16_t *q, const uint8_t *modality, float *logits, float2 *part,
                             DeviceError *err) {
  if (P.hkv == 4) {
    static std::atomic<uint64_t> attr{0};
    const cudaError_t e = once_per_device(attr, [] {
      return cudaFuncSetAttribute(score_narrow_tc_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(TcLayout<4>::kBytes));
    });
    if (e != cudaSuccess) return e;
    return launch_pdl(score_narrow_tc_kernel<4>, dim3(grid), dim3(tc_threads<4>()), TcLayout<4>::kBytes, stream,
                      kmap, P, q, modality, logits, part, err);
  } else {
    static std::atomic<uint64_t> attr{0};
    const cudaError_t e = once_per_device(attr, [] {
      return cudaFuncSetAttribute(score_narrow_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(TcLayout<2>::kBytes));
    });
    if (e != cudaSuccess) return e;
    return launch_pdl(score_narrow_tc_kernel<2>, dim3(grid), dim3(tc_threads<2>()), TcLayout<2>::kBytes, stream,
                      kmap, P, q, modality, logits, part, err);
  }
}

}  // namespace apack
