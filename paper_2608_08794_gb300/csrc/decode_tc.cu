// decode_tc.cu -- decode-step attention over a (compacted) KV cache on the tensor cores
// (Sec. 3.2, last sentence; App. G: the cost pruning shortens at every decode step).
//
//   out[b, h] = sum_j softmax_j(q[b, h] . k[j, g(h)] / sqrt(128)) v[j, g(h)]
//
// About one CTA per SM (each sequence gets CTAs in proportion to its length), all KV heads.  A
// stage is one KV head of one 128-key tile; the CTAs of a sequence claim its stages in order
// from a counter in the workspace (tile-major, heads within a tile), so that CTAs on SMs that
// stream faster take more of them and all finish together.  Each CTA folds every stage it
// claims into its running per-head state, so it still writes one partial per query head;
// which CTA takes which stage varies from call to call, and with it the last bits of the
// result.  The combine kernel resets the counter for the next call.  A stage's K rows and V
// rows (TMA boxes of 64 features x 1 head x 128 keys, 128-byte swizzle, 32 KB each) are
// separate items of a 6-slot shared-memory ring, loaded in the order K0 K1 V0 K2 V1 K3 V2 ...:
// the keys of a stage arrive one stage ahead of its values, so its logits and probabilities
// are ready when V lands, and each item holds its slot only until its own contraction is done
// (K: S, V: O^T).  The producer publishes each claimed stage (or the end of the claims) in a
// small ring of stage records with their own barriers, which every other role reads in order.
//   warp 0, one lane:  stage claims and TMA loads of the items
//   warp 1, one lane:  TMEM allocation; S = K q^T of every stage: keys as M = 128, the head
//                      group's <= 8 query rows (zero-padded) as N = 16; S[key][row] in TMEM
//   warp 6, one lane:  O^T += V^T P^T of every stage: features as M = 128 (V read as an MN-major
//                      operand straight from the stage), keys as K, N = 16 columns: the 8 rows'
//                      p split into a bf16 high part (columns 0..7) and the bf16 rounding of the
//                      remainder (8..15); O^T of each KV head stays in TMEM for the whole chunk.
//                      Two issuing warps, so that no stage's O^T waits for the next stage's data.
//   warps 2..5:        softmax, one key per thread (one TMEM lane): scaled logits, p = exp2(s - m)
//                      against a per-(head, row) reference maximum m that is only raised when a
//                      tile's logits exceed it by more than 2^8 (then O^T's columns of that row
//                      and the partial sums are rescaled once), p written as the bf16 pair into
//                      the head's P tile; at the end they read O^T back (one feature per thread).
// The result per query head is the CTA's partial (m, l = sum p, o = sum p v) in log2 units
// (m = -inf, l = 0, o = 0 for a head of which it claimed no stage),
// merged by the combine kernel with the CUDA-core kernel's partials' rules.  hi + lo carries p
// to about 2^-17 relative, so o matches fp32 arithmetic.  Every wait is bounded.
#include <cmath>

#include <cuda_bf16.h>

#include "decode_plan.cuh"
#include "internal.cuh"
#include "ptx.cuh"

namespace apack {
namespace {

constexpr int kDM = 128;                           // keys per tile (MMA M of S, K of O^T)
constexpr int kDN = 16;                            // MMA N: query rows (S), hi/lo rows (O^T)
constexpr int kDRows = 8;                          // rows handled (G <= 8)
constexpr int kDSlots = 6;
constexpr int kDHalf = kDM * 128;                  // 64 features x 128 keys x 2 B = 16 KB
constexpr int kDSlotBytes = 2 * kDHalf;            // K or V of one stage, two feature halves: 32 KB
constexpr int kDQHalf = kDN * 128;                 // 16 rows x 64 features x 2 B = 2 KB
constexpr int kDPBytes = 2 * kDN * 128;            // P^T of one head: 16 rows x 128 keys x 2 B = 4 KB
constexpr int kDSoftWarps = 4;
constexpr int kDPvWarp = 2 + kDSoftWarps;
constexpr int kDThreads = 32 * (3 + kDSoftWarps);
constexpr float kDLazy = 8.f;                      // the reference maximum lags by at most 2^8
constexpr uint32_t kDIdescS = idesc_bf16_f32(kDM, kDN);
constexpr uint32_t kDIdescO = idesc_bf16_f32(128, kDN) | (1u << 15);   // A (V^T) MN-major
constexpr uint32_t kDTmemCols = 128;               // S [2][16] at 0, O^T of head h at 32 + 16 h
constexpr int kDInfo = 8;                          // stage records in flight (the producer leads by <= 5)

struct __align__(8) DBars {
  uint64_t full[kDSlots], empty[kDSlots], s_full[2], s_empty[2], drain[2];   // drain: per issuing warp
  uint64_t p_full[4], p_empty[4];                  // one pair per KV head: their phases are its stages
  uint64_t info_full[kDInfo];                      // stage record n % kDInfo written (phase n / kDInfo)
  volatile int32_t info[kDInfo];                   // claimed unit (tile * HKV + head), or -1: no more
  uint32_t tmem_base;
  volatile int32_t abort;
};

template <int HKV>
struct DLay {
  static constexpr uint32_t kOffQ = kDSlots * kDSlotBytes;                      // 1024-aligned
  static constexpr uint32_t kOffP = kOffQ + HKV * 2 * kDQHalf;                   // [HKV] P^T tiles, 1024-aligned
  static constexpr uint32_t kOffT = kOffP + HKV * kDPBytes;                      // tile maxima [2][4][8]
  static constexpr uint32_t kOffM = kOffT + 2 * kDSoftWarps * kDRows * 4;        // reference max [2][HKV][8]
  static constexpr uint32_t kOffBars = (kOffM + 2 * HKV * kDRows * 4 + 7) & ~7u;
  static constexpr uint32_t kBytes = kOffBars + 512;
};
static_assert(sizeof(DBars) <= 512, "barrier block");

__device__ __forceinline__ bool d_wait(uint64_t *bar, uint32_t parity, DBars *bars, DeviceError *err, int where) {
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

// Named barrier over `count` threads that also ORs a predicate across them.
__device__ __forceinline__ bool bar_red_or(uint32_t id, uint32_t count, bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, %2, %3, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(v)), "r"(id), "r"(count)
      : "memory");
  return r != 0;
}

// byte offset of element (row, key) in a 16-row x 128-key bf16 K-major tile, 128-byte swizzle
__device__ __forceinline__ uint32_t p_off(int row, int key) {
  const int half = key >> 6, ch = (key & 63) >> 3;
  return half * 2048 + (row >> 3) * 1024 + (row & 7) * 128 + ((ch ^ (row & 7)) << 4) + (key & 7) * 2;
}

// Load order of the ring's items: K0, K1, V0, K2, V1, K3, V2, ...  With N claimed stages the
// position of K(N) carries no load (the end of the claims) and V(N-1) is the last item.
__device__ __forceinline__ int item_of_k(int n) { return n == 0 ? 0 : 2 * n - 1; }
__device__ __forceinline__ int item_of_v(int n) { return 2 * n + 2; }
__device__ __forceinline__ void item_stage(int i, bool *is_v, int *n) {
  if (i == 0) { *is_v = false; *n = 0; }
  else if (i & 1) { *is_v = false; *n = (i + 1) >> 1; }
  else { *is_v = true; *n = (i >> 1) - 1; }
}

template <int HKV>
__global__ void __launch_bounds__(kDThreads, 1)
    decode_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const __grid_constant__ DecPlan plan, const uint16_t *__restrict__ q, float *__restrict__ opart,
                     float2 *__restrict__ mlpart, unsigned int *claims, DeviceError *err) {
  using Lay = DLay<HKV>;
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");   // the combine may be scheduled
  extern __shared__ __align__(1024) uint8_t smem[];
  if ((smem_u32(smem) & 1023u) != 0) {
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 90);
    return;
  }
  uint8_t *ring = smem;
  uint8_t *qs = smem + Lay::kOffQ;
  uint8_t *ps = smem + Lay::kOffP;
  float *tmax = reinterpret_cast<float *>(smem + Lay::kOffT);
  float *msm = reinterpret_cast<float *>(smem + Lay::kOffM);
  DBars *bars = reinterpret_cast<DBars *>(smem + Lay::kOffBars);
  const int c = blockIdx.x;
  const int s = find_chunk_seq(plan, c);
  const DecSeq &sq = plan.seq[s];
  const int G = plan.group;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int units = (sq.len + kDM - 1) / kDM * HKV;   // the sequence's stages

  if (threadIdx.x == 0) {
    for (int i = 0; i < kDSlots; ++i) {
      mbar_init(&bars->full[i], 1);
      mbar_init(&bars->empty[i], 1);                // the commit after the item's MMAs
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->s_full[i], 1);
      mbar_init(&bars->s_empty[i], kDSoftWarps);
    }
    for (int h = 0; h < HKV; ++h) {
      mbar_init(&bars->p_full[h], kDSoftWarps);
      mbar_init(&bars->p_empty[h], 1);
    }
    mbar_init(&bars->drain[0], 1);
    mbar_init(&bars->drain[1], 1);
    for (int i = 0; i < kDInfo; ++i) mbar_init(&bars->info_full[i], 1);
    bars->abort = 0;
    for (int i = 0; i < 2 * HKV * kDRows; ++i) msm[i] = -INFINITY;
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(&bars->tmem_base, kDTmemCols);
    tc_fence_before();
  }
  // Launched as a programmatic dependent: the set-up above runs beside the previous launch on
  // the stream; q, the cache and the partials (which the previous call's combine reads) are
  // touched only once that launch has completed.
  asm volatile("griddepcontrol.wait;" ::: "memory");
  // query tiles: rows j < G of head group h, 128-byte swizzled K-major layout
  for (int idx = threadIdx.x; idx < HKV * kDN * 16; idx += kDThreads) {
    const int h = idx / (kDN * 16), rem = idx % (kDN * 16);
    const int row = rem / 16, ch = rem % 16;
    const int half = ch >> 3, cc = ch & 7;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (row < G)
      v = __ldg(reinterpret_cast<const uint4 *>(q + (static_cast<int64_t>(s) * plan.hq + h * G + row) * 128) + ch);
    *reinterpret_cast<uint4 *>(qs + h * 2 * kDQHalf + half * kDQHalf + (row >> 3) * 1024 + (row & 7) * 128 +
                               ((cc ^ (row & 7)) << 4)) = v;
  }
  fence_proxy_async_smem();
  __syncthreads();
  tc_fence_after();

  float l_run[HKV][kDRows];                        // softmax threads: partial sums of their keys
#pragma unroll
  for (int h = 0; h < HKV; ++h)
#pragma unroll
    for (int j = 0; j < kDRows; ++j) l_run[h][j] = 0.f;
  bool stop = false;
  uint32_t par = 0, seen = 0;                      // softmax threads, per KV head: stage-count parity, any stage

  if (warp == 0) {
    // ------------------------------------------------------------ claims and TMA producer
    if (lane == 0) {
      tma_prefetch_desc(&kmap);
      tma_prefetch_desc(&vmap);
      // claims run two stages ahead of the loads (an atomic's round trip is about a stage's
      // time); one thread's claims on one counter return increasing units
      unsigned int *claim = claims + s;
      int next = static_cast<int>(atomicAdd(claim, 1u));   // stage 0's unit
      int next2 = static_cast<int>(atomicAdd(claim, 1u));  // stage 1's
      int unit[2] = {0, 0};                       // units of the last two claimed stages (by n & 1)
      int n_end = -1;                             // the number of claimed stages, once known
      int last = -1;                              // the last item issued with a load
      bool pend[kDSlots] = {};
      uint32_t pend_par[kDSlots] = {};
      for (int i = 0;; ++i) {
        bool is_v;
        int n;
        item_stage(i, &is_v, &n);
        if (n_end >= 0 && (!is_v || n >= n_end)) break;
        const int slot = i % kDSlots;
        if (!is_v) {
          // publish stage n's record (its unit, or the end of the claims) before its K load
          const int u = next;
          const int r = n % kDInfo;
          if (u >= units) {
            bars->info[r] = -1;
            mbar_arrive(&bars->info_full[r]);
            n_end = n;
            continue;                              // no load: V(n - 1) is the last item
          }
          next = next2;
          next2 = static_cast<int>(atomicAdd(claim, 1u));  // stage n + 2's unit
          unit[n & 1] = u;
          bars->info[r] = u;
          mbar_arrive(&bars->info_full[r]);
        }
        if (i >= kDSlots && !d_wait(&bars->empty[slot], ((i / kDSlots) - 1) & 1u, bars, err, 91)) break;
        const int u = unit[n & 1];
        const int t = u / HKV, h = u % HKV;
        uint8_t *dst = ring + slot * kDSlotBytes;
        const CUtensorMap *map = is_v ? &vmap : &kmap;
        mbar_arrive_expect_tx(&bars->full[slot], kDSlotBytes);
        const int key0 = sq.t0 + t * kDM;
        tma_load_3d(dst, map, &bars->full[slot], 0, h, key0);
        tma_load_3d(dst + kDHalf, map, &bars->full[slot], 64, h, key0);
        pend[slot] = true;
        pend_par[slot] = (i / kDSlots) & 1u;
        last = i;
      }
      if (bars->abort) {
        for (int i = 0; i < kDSlots; ++i)
          if (pend[i]) mbar_wait(&bars->full[i], pend_par[i], kWaitLimitNs / 4);
      } else {
        // every loaded item's slot is released by a commit after its MMAs; the last loaded item
        // of each slot is awaited here (earlier ones were, before their slots were reloaded), so
        // that no commit arrives after the CTA has left.  The end marker loads nothing and no
        // item after it shares its slot; the kDSlots + 2 latest positions cover every slot.
        const int k_end = n_end >= 0 ? item_of_k(n_end) : -1;
        uint32_t waited = 0;
        for (int k = last; k >= 0 && k >= last - kDSlots - 1; --k) {
          const int sl = k % kDSlots;
          if (k == k_end || ((waited >> sl) & 1u)) continue;
          waited |= 1u << sl;
          d_wait(&bars->empty[sl], (k / kDSlots) & 1u, bars, err, 89);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ S issuer
    if (lane == 0) {
      const uint32_t tmem = bars->tmem_base;
      const uint32_t q_base = smem_u32(qs);
      bool issued = false;
      for (int n = 0;; ++n) {
        const int r = n % kDInfo;
        if (!d_wait(&bars->info_full[r], (n / kDInfo) & 1u, bars, err, 99)) break;
        const int u = bars->info[r];
        if (u < 0) break;
        const int item = item_of_k(n), slot = item % kDSlots, buf = n & 1, h = u % HKV;
        if (n >= 2 && !d_wait(&bars->s_empty[buf], ((n >> 1) - 1) & 1u, bars, err, 92)) break;
        if (!d_wait(&bars->full[slot], (item / kDSlots) & 1u, bars, err, 93)) break;
        tc_fence_after();
        // K (two 64-feature halves) against the head group's query rows, 16 features per MMA
        const uint32_t a_base = smem_u32(ring + slot * kDSlotBytes);
        const uint32_t b_base = q_base + h * 2 * kDQHalf;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t ao = (kk >> 2) * kDHalf + (kk & 3) * 32;
          const uint32_t bo = (kk >> 2) * kDQHalf + (kk & 3) * 32;
          tc_mma_bf16(tmem + buf * kDN, smem_desc_sw128(a_base + ao), smem_desc_sw128(b_base + bo), kDIdescS,
                      kk > 0 ? 1u : 0u);
        }
        tc_commit(&bars->s_full[buf]);
        tc_commit(&bars->empty[slot]);              // K is free once S is done
        issued = true;
      }
      if (issued) {                                 // every MMA of this thread done before teardown
        tc_commit(&bars->drain[0]);
        mbar_wait(&bars->drain[0], 0, kWaitLimitNs / 4);
      }
    }
  } else if (warp == kDPvWarp) {
    // ------------------------------------------------------------ O^T issuer
    if (lane == 0) {
      const uint32_t tmem = bars->tmem_base;
      const uint32_t p_base = smem_u32(ps);
      uint32_t opar = 0, oseen = 0;                 // per KV head: stage-count parity, any stage
      for (int n = 0;; ++n) {
        const int r = n % kDInfo;
        if (!d_wait(&bars->info_full[r], (n / kDInfo) & 1u, bars, err, 99)) break;
        const int u = bars->info[r];
        if (u < 0) break;
        const int item = item_of_v(n), slot = item % kDSlots, h = u % HKV;
        if (!d_wait(&bars->p_full[h], (opar >> h) & 1u, bars, err, 94)) break;
        if (!d_wait(&bars->full[slot], (item / kDSlots) & 1u, bars, err, 98)) break;
        tc_fence_after();
        // O^T[feature][col] += sum_key V[key][feature] P^T[col][key]: 16 keys per MMA
        const uint32_t v_base = smem_u32(ring + slot * kDSlotBytes);
        const uint32_t b_base = p_base + h * kDPBytes;
        const bool acc = (oseen >> h) & 1u;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint32_t bo = (kk >> 2) * (kDPBytes / 2) + (kk & 3) * 32;
          tc_mma_bf16(tmem + 32 + h * kDN, smem_desc_sw128_mn(v_base + kk * 2048, kDHalf, 1024),
                      smem_desc_sw128(b_base + bo), kDIdescO, (acc || kk > 0) ? 1u : 0u);
        }
        tc_commit(&bars->p_empty[h]);
        tc_commit(&bars->empty[slot]);
        opar ^= 1u << h;
        oseen |= 1u << h;
      }
      if (oseen) {
        tc_commit(&bars->drain[1]);
        mbar_wait(&bars->drain[1], 0, kWaitLimitNs / 4);
      }
    }
  } else {
    // ------------------------------------------------------------ softmax, one key per thread (warps 2..5)
    const int sw = warp - 2;
    const int quad = warp & 3;                       // TMEM lanes 32 * (warp % 4) ..
    const int kt = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const float c2 = plan.scale2;
    const bool odd = lane & 1;
    for (int n = 0;; ++n) {
      // the stage's record; the four warps leave together, at a barrier, at the end of the
      // claims or when a wait gave up
      const int r = n % kDInfo;
      bool ok = __all_sync(0xffffffffu, d_wait(&bars->info_full[r], (n / kDInfo) & 1u, bars, err, 99));
      const int u = ok ? bars->info[r] : -1;
      if (bar_red_or(1, kDSoftWarps * 32, !ok || u < 0)) {
        stop = bar_red_or(1, kDSoftWarps * 32, !ok);
        break;
      }
      const int t = u / HKV, h = u % HKV, buf = n & 1;
      const bool hseen = (seen >> h) & 1u;
      const uint32_t hpar = (par >> h) & 1u;
      // every wait of the stage comes first; the group leaves only together, at a barrier
      ok = __all_sync(0xffffffffu, d_wait(&bars->s_full[buf], (n >> 1) & 1u, bars, err, 95));
      if (ok && hseen)   // the head's previous O^T MMAs are done: its P tile and O^T are free
        ok = __all_sync(0xffffffffu, d_wait(&bars->p_empty[h], hpar ^ 1u, bars, err, 96));
      const int key = t * kDM + kt;
      const bool valid = key < sq.len;
      const float *m_old = msm + (hpar ^ 1u) * HKV * kDRows + h * kDRows;
      float *m_new = msm + hpar * HKV * kDRows + h * kDRows;
      float x[kDRows], m[kDRows];
      bool raise = false;
#pragma unroll
      for (int j = 0; j < kDRows; ++j) {
        x[j] = -INFINITY;
        m[j] = m_old[j];
      }
      if (ok) {
        tc_fence_after();
        uint32_t rr[8];
        tmem_ld8_wait(bars->tmem_base + lane_off + buf * kDN, rr);
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->s_empty[buf]);
#pragma unroll
        for (int j = 0; j < kDRows; ++j) {
          x[j] = (valid && j < G) ? __uint_as_float(rr[j]) * c2 : -INFINITY;
          raise |= x[j] > m[j] + kDLazy;           // also every finite logit against -inf
        }
      }
      const bool bad = !ok || bars->abort;
      if (bar_red_or(1, kDSoftWarps * 32, bad || raise)) {
        // slow path (the head's first stage, a new maximum, or an abort): the tile's row maxima
        float *tm = tmax + buf * kDSoftWarps * kDRows;
#pragma unroll
        for (int j = 0; j < kDRows; ++j) {
          float wm = x[j];
#pragma unroll
          for (int off = 16; off > 0; off >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, off));
          if (lane == 0) tm[sw * kDRows + j] = wm;
        }
        if (bar_red_or(1, kDSoftWarps * 32, bad)) {
          stop = true;
          break;
        }
        float f[kDRows];
        bool any = false;
#pragma unroll
        for (int j = 0; j < kDRows; ++j) {
          const float mt = fmaxf(fmaxf(tm[j], tm[kDRows + j]), fmaxf(tm[2 * kDRows + j], tm[3 * kDRows + j]));
          f[j] = 1.f;
          if (mt > m[j] + kDLazy) {               // the same decision in every thread
            f[j] = m[j] == -INFINITY ? 0.f : ex2_approx(m[j] - mt);
            m[j] = mt;
            any = true;
          }
        }
#pragma unroll
        for (int hh = 0; hh < HKV; ++hh)            // register-resident sums: head selected by predicate
          if (hh == h)
#pragma unroll
            for (int j = 0; j < kDRows; ++j) l_run[hh][j] *= f[j];
        if (any && hseen) {
          // rescale the head's O^T columns (this thread's feature kt): hi and lo alike
          uint32_t o[16];
          tc_fence_after();
          tmem_ld16_wait(bars->tmem_base + lane_off + 32 + h * kDN, o);
#pragma unroll
          for (int j = 0; j < kDRows; ++j) {
            o[j] = __float_as_uint(__uint_as_float(o[j]) * f[j]);
            o[j + 8] = __float_as_uint(__uint_as_float(o[j + 8]) * f[j]);
          }
          tmem_st16_wait(bars->tmem_base + lane_off + 32 + h * kDN, o);
          tc_fence_before();
        }
      }
      // p = exp2(s - m) as a bf16 pair into the head's P^T tile; the even lane of a key pair
      // writes the high parts of both keys, the odd lane the low parts (rows rotated by 4 so
      // that the two halves of the warp hit different banks)
      float pv[kDRows];
      uint32_t hl[kDRows];                         // (hi | lo << 16) of this key, per row
#pragma unroll
      for (int j = 0; j < kDRows; ++j) {
        pv[j] = x[j] == -INFINITY ? 0.f : ex2_approx(x[j] - m[j]);
        const __nv_bfloat16 hi = __float2bfloat16_rn(pv[j]);
        const __nv_bfloat16 lo = __float2bfloat16_rn(pv[j] - __bfloat162float(hi));
        hl[j] = static_cast<uint32_t>(__bfloat16_as_ushort(hi)) |
                (static_cast<uint32_t>(__bfloat16_as_ushort(lo)) << 16);
      }
#pragma unroll
      for (int hh = 0; hh < HKV; ++hh)
        if (hh == h)
#pragma unroll
          for (int j = 0; j < kDRows; ++j) l_run[hh][j] += pv[j];
      uint8_t *pt = ps + h * kDPBytes;
#pragma unroll
      for (int j = 0; j < kDRows; ++j) {
        const int jl = (j + 4) & 7;
        const uint32_t send = odd ? (hl[j] & 0xFFFFu) : (hl[jl] >> 16);
        const uint32_t recv = __shfl_xor_sync(0xffffffffu, send, 1);
        if (!odd)   // keys kt, kt + 1: high parts of row j
          *reinterpret_cast<uint32_t *>(pt + p_off(j, kt)) = (hl[j] & 0xFFFFu) | (recv << 16);
        else        // keys kt - 1, kt: low parts of row jl
          *reinterpret_cast<uint32_t *>(pt + p_off(8 + jl, kt - 1)) = recv | (hl[jl] & 0xFFFF0000u);
      }
      if (kt == 0)
#pragma unroll
        for (int j = 0; j < kDRows; ++j) m_new[j] = m[j];
      fence_proxy_async_smem();                    // the P tile is read by the tensor cores
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->p_full[h]);
      par ^= 1u << h;
      seen |= 1u << h;
    }
    // each head's last O^T MMAs must be complete before O^T is read
    if (!stop)
#pragma unroll
      for (int h = 0; h < HKV; ++h)
        if (((seen >> h) & 1u) &&
            !__all_sync(0xffffffffu, d_wait(&bars->p_empty[h], ((par >> h) & 1u) ^ 1u, bars, err, 97)))
          break;
  }

  // ---------------------------------------------------------------- epilogue and teardown
  tc_fence_before();
  __syncthreads();                              // every stage consumed: the ring is free
  tc_fence_after();
  const bool ok = !bars->abort;
  float *lsum = reinterpret_cast<float *>(ring);                         // [HKV * 8][128 keys]
  float *mrow = lsum + kDM * HKV * kDRows;                                // [HKV][8]
  if (ok && warp >= 2 && warp < kDPvWarp) {
    const int quad = warp & 3, kt = quad * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
#pragma unroll
    for (int h = 0; h < HKV; ++h) {
      uint32_t o[16];
#pragma unroll
      for (int j = 0; j < 16; ++j) o[j] = 0u;
      if ((seen >> h) & 1u)                      // uniform over the softmax warps
        tmem_ld16_wait(bars->tmem_base + lane_off + 32 + h * kDN, o);
#pragma unroll
      for (int j = 0; j < kDRows; ++j)           // feature kt of row j: high plus low part
        if (j < G)
          opart[(static_cast<int64_t>(c) * plan.hq + h * G + j) * 128 + kt] =
              __uint_as_float(o[j]) + __uint_as_float(o[j + 8]);
#pragma unroll
      for (int j = 0; j < kDRows; ++j) lsum[(h * kDRows + j) * kDM + kt] = l_run[h][j];
    }
    if (kt == 0)   // the reference maximum of each head's last stage (-inf: no stage)
#pragma unroll
      for (int h = 0; h < HKV; ++h)
#pragma unroll
        for (int j = 0; j < kDRows; ++j)
          mrow[h * kDRows + j] = ((seen >> h) & 1u)
                                     ? msm[(((par >> h) & 1u) ^ 1u) * HKV * kDRows + h * kDRows + j]
                                     : -INFINITY;
  }
  tc_fence_before();
  __syncthreads();
  if (ok) {
    // one warp per (head, row): the 128 partial sums in a fixed order
    for (int e = warp; e < HKV * G; e += kDThreads / 32) {
      const int h = e / G, j = e % G;
      const float4 l4 = *reinterpret_cast<const float4 *>(lsum + (h * kDRows + j) * kDM + lane * 4);
      float l = (l4.x + l4.y) + (l4.z + l4.w);
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) l += __shfl_xor_sync(0xffffffffu, l, off);
      if (lane == 0) mlpart[static_cast<int64_t>(c) * plan.hq + h * G + j] = make_float2(mrow[h * kDRows + j], l);
    }
  }
  tc_fence_after();
  if (warp == 1) tmem_dealloc(bars->tmem_base, kDTmemCols);
}

}  // namespace

cudaError_t launch_decode_tc(int grid, cudaStream_t stream, const CUtensorMap &kmap, const CUtensorMap &vmap,
                             const DecPlan &P, const uint16_t *q, float *opart, float2 *mlpart, unsigned int *claims,
                             DeviceError *err) {
  if (P.hkv == 4) {
    static std::atomic<uint64_t> attr{0};
    const cudaError_t e = once_per_device(attr, [] {
      return cudaFuncSetAttribute(decode_tc_kernel<4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(DLay<4>::kBytes));
    });
    if (e != cudaSuccess) return e;
    return launch_pdl(decode_tc_kernel<4>, dim3(grid), dim3(kDThreads), DLay<4>::kBytes, stream, kmap, vmap, P, q,
                      opart, mlpart, claims, err);
  } else {
    static std::atomic<uint64_t> attr{0};
    const cudaError_t e = once_per_device(attr, [] {
      return cudaFuncSetAttribute(decode_tc_kernel<2>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(DLay<2>::kBytes));
    });
    if (e != cudaSuccess) return e;
    return launch_pdl(decode_tc_kernel<2>, dim3(grid), dim3(kDThreads), DLay<2>::kBytes, stream, kmap, vmap, P, q,
                      opart, mlpart, claims, err);
  }
}

}  // namespace apack
