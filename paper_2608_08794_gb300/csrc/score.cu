// score.cu -- relevance scores of Eq. inner_score (Sec. 3.2) on the tcgen05 tensor cores.
//
// I_i = 1/(Hq n_q) sum_h sum_r softmax_{j in S}(q_{r,h} . k_{j,g(h)} / sqrt(D))_i
//
// The softmax normaliser of every (query row, head) needs all keys of S before
// any per-key average can be formed, so the scores take two passes over K:
//
//  pass 1 (row statistics): D[row][key] = Q . K_block^T with query rows in TMEM
//     lanes; each epilogue thread owns one row and keeps an online (reference,
//     sum of exp2) over its keys.  Keys are split across CTAs; each (split, row)
//     writes a partial pair.
//  merge: per row, the partials combine into a log2-domain normaliser
//     lse2 = log2 sum_j 2^(x_j log2(e)/sqrt(D)), stored negated per 128-row chunk.
//  pass 2 (column sums): D[key][row] = K . Q_chunk^T with keys in TMEM lanes;
//     each thread owns one key and sums 2^(x c - lse2[row]) over the rows of one
//     KV head group; a final pass adds the Hkv group sums in a fixed order and
//     scales by 1/(Hq n_q).  No atomics anywhere: scores are deterministic.
//
// Query rows are first repacked per KV head g into linear rows rho = token * G + j
// (query head g*G + j), padded to a multiple of 256, so that tiles hold no holes.
//
// Both passes: A operand = two 128-row tiles (256 rows of Q in pass 1, 256 keys
// in pass 2), B operand = a 128-row tile streamed through a 3-stage TMA ring;
// each B tile feeds two M=128 x N=128 MMAs, one per A tile, into one of two
// 256-column TMEM accumulators.  Warp 0 issues TMA, warp 1 owns TMEM and
// issues tcgen05.mma, warps 2..17 are four epilogue warpgroups, warpgroup
// (t, h) reading columns h*64.. of A tile t's accumulator; the two halves of
// a row (pass 1) or key (pass 2) are combined once per work unit through
// shared memory.  Operands sit in 128-byte swizzled shared memory.
// Persistent CTAs, one per SM (the shared-memory footprint allows one).
#include <cmath>
#include <cstdio>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kThreads = 576;          // warp 0: TMA, warp 1: MMA, warps 2..17: epilogue
constexpr int kEpiWarps = 16;          // four warpgroups: (A tile t, column half h) each
constexpr uint32_t kTmemCols = 512;    // 2 accumulators x 2 tiles x 128 fp32 columns
constexpr int kAStages = 2, kBStages = 3;
constexpr uint32_t kARows = 256, kBRows = 128;
constexpr uint32_t kABytes = kARows * 256;     // 256 rows x 128 bf16
constexpr uint32_t kBBytes = kBRows * 256;     // 128 rows x 128 bf16
constexpr uint32_t kAHalf = kARows * 128;      // second 64-element K half of A
constexpr uint32_t kBHalf = kBRows * 128;      // ... of B
constexpr uint32_t kATile = 128 * 128;         // second 128-row tile within an A half
constexpr uint32_t kIdesc = idesc_bf16_f32(128, 128);
constexpr int kKeysPerBlock1 = kBRows;         // pass 1: keys per B tile
constexpr int kKeysPerUnit2 = kARows;          // pass 2: keys per work unit (two tiles)

struct SeqPlan {
  int32_t t0, len;        // token range of the sequence in the packed batch
  int32_t q_off, n_q;     // query tokens in packed Q
  int32_t qp_base;        // first packed row of head group 0; group g starts at qp_base + g * rows_pad
  int32_t rows_pad;       // G * n_q rounded up to a multiple of 256
  int32_t unit_begin;     // first work unit of this sequence in the launch
  int32_t bps;            // pass 1: key blocks per split
  int32_t n_split;        // pass 1: splits
  int32_t chunk_base;     // index of this sequence's first normaliser chunk
};

struct ScorePlan {
  int32_t nseq;
  int32_t total_units;
  int32_t hq, hkv, group;
  int32_t total_qrows;     // sum n_q over the whole batch
  int32_t total_tokens;    // T
  int32_t causal;          // APACK_SOFTMAX_CAUSAL_ROW: rows see every token up to their own position
  float scale2;            // log2(e) / sqrt(D)
  SeqPlan seq[kSeqsPerLaunch];
};

struct __align__(8) Bars {
  uint64_t a_full[kAStages], a_empty[kAStages], b_full[kBStages], b_empty[kBStages];
  uint64_t acc_full[2], acc_empty[2], drain;
  uint64_t l_empty[kBStages];       // pass 2: normaliser slot released by the epilogue
  uint64_t comb_full[2], comb_empty[2];   // pass 2, per key tile: column half 1 -> half 0 hand-off
  uint32_t tmem_base;
  volatile int32_t abort;
};

// Shared memory: [A x2][B x3][-lse2 x3 (pass 2)][combine 2 x 128 float (pass 2)][Bars].
// The dynamic shared window is declared 1024-byte aligned (the 128-byte swizzle
// atoms of the operand tiles need it); the kernels verify it before any use.
constexpr uint32_t kOffA = 0;
constexpr uint32_t kOffB = kAStages * kABytes;
constexpr uint32_t kOffL = kOffB + kBStages * kBBytes;
constexpr uint32_t kOffC = kOffL + kBStages * kBRows * sizeof(float);
constexpr uint32_t kOffBars = kOffC + 2 * 128 * sizeof(float);
constexpr uint32_t kSmemBytes = kOffBars + 256;
static_assert(kSmemBytes <= 232448, "shared memory budget");

__device__ __forceinline__ int find_seq(const ScorePlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit_begin <= u) ++s;
  return s;
}

__device__ __forceinline__ bool is_mm(uint8_t m) { return m == APACK_MOD_AUDIO || m == APACK_MOD_VISUAL; }

__host__ __device__ __forceinline__ int n_pairs(const SeqPlan &sp) { return sp.rows_pad / 256; }
__host__ __device__ __forceinline__ int n_chunks(const SeqPlan &sp, int G) { return (G * sp.n_q + 127) / 128; }
__host__ __device__ __forceinline__ int n_keypairs(const SeqPlan &sp) { return (sp.len + 255) / 256; }

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

// True when the dynamic shared window has the 1024-byte alignment the operand tiles need.
__device__ __forceinline__ bool smem_aligned(const uint8_t *smem) { return (smem_u32(smem) & 1023u) == 0; }

__device__ void init_common(uint8_t *smem, Bars *bars, int warp) {
  // Zero the operand buffers so that MMA rows no TMA box writes stay finite.
  for (uint32_t i = threadIdx.x; i < kOffL / 16; i += blockDim.x)
    reinterpret_cast<uint4 *>(smem)[i] = make_uint4(0, 0, 0, 0);
  if (threadIdx.x == 0) {
    for (int i = 0; i < kAStages; ++i) {
      mbar_init(&bars->a_full[i], 1);
      mbar_init(&bars->a_empty[i], 1);
    }
    for (int i = 0; i < kBStages; ++i) {
      mbar_init(&bars->b_full[i], 1);
      mbar_init(&bars->b_empty[i], 1);
      mbar_init(&bars->l_empty[i], kEpiWarps);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], kEpiWarps);
      mbar_init(&bars->comb_full[i], 128);
      mbar_init(&bars->comb_empty[i], 128);
    }
    mbar_init(&bars->drain, 1);
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
}

// Teardown: after an abort the MMA thread makes sure no MMA is in flight; then TMEM is freed.
__device__ void finish_common(Bars *bars, int warp, bool mma_thread) {
  if (mma_thread && bars->abort) {
    tc_commit(&bars->drain);
    mbar_wait(&bars->drain, 0, kWaitLimitNs / 4);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(bars->tmem_base, kTmemCols);
}

// Waits (bounded, ignoring the abort flag) for TMA loads that were issued
// but never consumed, so that no copy lands in shared memory after exit.
__device__ void drain_loads(uint64_t *full, const bool *pending, const uint32_t *parity, int n) {
  for (int i = 0; i < n; ++i)
    if (pending[i]) mbar_wait(&full[i], parity[i], kWaitLimitNs / 4);
}

// Issues the two MMAs of one B tile (one per A tile) into accumulator `ci`.
__device__ __forceinline__ void issue_mma_pair(uint32_t tmem, int ci, uint32_t a_base, uint32_t b_base, int ntiles) {
  for (int t = 0; t < ntiles; ++t) {
#pragma unroll
    for (int kk = 0; kk < 8; ++kk) {
      const uint32_t ao = (kk >> 2) * kAHalf + t * kATile + (kk & 3) * 32;
      const uint32_t bo = (kk >> 2) * kBHalf + (kk & 3) * 32;
      tc_mma_bf16(tmem + ci * 256 + t * 128, smem_desc_sw128(a_base + ao), smem_desc_sw128(b_base + bo), kIdesc,
                  kk > 0 ? 1u : 0u);
    }
  }
}

// ------------------------------------------------------------------ pass 1
struct Unit1 {
  int s, g, qp, b0, b1, split, ntiles;
};

__device__ __forceinline__ Unit1 decode_unit1(const ScorePlan &p, int u) {
  Unit1 w;
  w.s = find_seq(p, u);
  const SeqPlan &sp = p.seq[w.s];
  const int local = u - sp.unit_begin;
  const int np = n_pairs(sp);
  w.qp = local % np;
  const int pg = local / np;
  w.g = pg % p.hkv;
  w.split = pg / p.hkv;
  const int nb = (sp.len + kKeysPerBlock1 - 1) / kKeysPerBlock1;
  w.b0 = w.split * sp.bps;
  w.b1 = min(nb, w.b0 + sp.bps);
  w.ntiles = p.group * sp.n_q - w.qp * 256 > 128 ? 2 : 1;
  return w;
}

// Online (reference, sum) update with 32 logits in log2 units: the reference
// is only raised when a value exceeds it by 2^64 (sum overflow check), which
// keeps the max computation off the common path.  Four independent partial
// sums keep the add chain short.
template <int OFF>
__device__ __forceinline__ void online_chunk(const uint32_t (&r)[64], uint32_t mask, float c2, float &m,
                                             float &sum) {
  if (mask == 0u) return;
  if (m == -INFINITY) {
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if ((mask >> i) & 1u) mx = fmaxf(mx, __uint_as_float(r[OFF + i]));
    m = mx * c2;
  }
  float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  const float2 cc = make_float2(c2, c2), nm = make_float2(-m, -m);
  if (mask == 0xffffffffu) {
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      const float2 y = ffma2(make_float2(__uint_as_float(r[OFF + i]), __uint_as_float(r[OFF + i + 1])), cc, nm);
      a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(ex2_approx(y.x), ex2_approx(y.y)));
    }
  } else {
#pragma unroll
    for (int i = 0; i < 32; i += 2) {
      const float2 y = ffma2(make_float2(__uint_as_float(r[OFF + i]), __uint_as_float(r[OFF + i + 1])), cc, nm);
      a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(((mask >> i) & 1u) ? ex2_approx(y.x) : 0.f,
                                                           ((mask >> (i + 1)) & 1u) ? ex2_approx(y.y) : 0.f));
    }
  }
  const float2 s01 = fadd2(a[0], a[1]), s23 = fadd2(a[2], a[3]);
  const float2 s4 = fadd2(s01, s23);
  float t = s4.x + s4.y;
  if (!(t <= 1.8446744e19f)) {   // a value exceeded the reference by more than 2^64 (or inf): rescale
    float mx = -INFINITY;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if ((mask >> i) & 1u) mx = fmaxf(mx, __uint_as_float(r[OFF + i]));
    mx *= c2;
    sum *= ex2_approx(m - mx);
    m = mx;
    t = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
      if ((mask >> i) & 1u) t += ex2_approx(fmaf(__uint_as_float(r[OFF + i]), c2, -m));
  }
  sum += t;
}

template <bool CAUSAL>
__global__ void __launch_bounds__(kThreads, 1)
    score_rowstats_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                          const __grid_constant__ ScorePlan plan, const uint8_t *__restrict__ modality,
                          float2 *__restrict__ part, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (!smem_aligned(smem)) {
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 10);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  init_common(smem, bars, warp);
  const int G = plan.group;

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[kBStages] = {}, apend[kAStages] = {};
      uint32_t pend_par[kBStages] = {}, apend_par[kAStages] = {};
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        const Unit1 w = decode_unit1(plan, u);
        const SeqPlan &sp = plan.seq[w.s];
        if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, err, 11)) { ok = false; break; }
        uint8_t *A = smem + kOffA + ai * kABytes;
        mbar_arrive_expect_tx(&bars->a_full[ai], kABytes);
        const int arow = sp.qp_base + w.g * sp.rows_pad + w.qp * 256;
        tma_load_3d(A, &qmap, &bars->a_full[ai], 0, 0, arow);
        tma_load_3d(A + kAHalf, &qmap, &bars->a_full[ai], 64, 0, arow);
        apend[ai] = true;
        apend_par[ai] = aph;
        for (int b = w.b0; b < w.b1; ++b) {
          if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, err, 12)) { ok = false; break; }
          uint8_t *B = smem + kOffB + bi * kBBytes;
          mbar_arrive_expect_tx(&bars->b_full[bi], kBBytes);
          const int key0 = sp.t0 + b * kKeysPerBlock1;
          tma_load_3d(B, &kmap, &bars->b_full[bi], 0, w.g, key0);
          tma_load_3d(B + kBHalf, &kmap, &bars->b_full[bi], 64, w.g, key0);
          pend[bi] = true;
          pend_par[bi] = bph;
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
        }
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
      if (!ok) {
        drain_loads(bars->b_full, pend, pend_par, kBStages);
        drain_loads(bars->a_full, apend, apend_par, kAStages);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        const Unit1 w = decode_unit1(plan, u);
        if (!wait_or_abort(&bars->a_full[ai], aph, bars, err, 13)) { ok = false; break; }
        const uint32_t a_base = smem_u32(smem + kOffA + ai * kABytes);
        for (int b = w.b0; b < w.b1; ++b) {
          if (!wait_or_abort(&bars->b_full[bi], bph, bars, err, 14)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, err, 15)) { ok = false; break; }
          tc_fence_after();
          issue_mma_pair(tmem, ci, a_base, smem_u32(smem + kOffB + bi * kBBytes), w.ntiles);
          tc_commit(&bars->b_empty[bi]);
          tc_commit(&bars->acc_full[ci]);
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
        if (!ok) break;
        tc_commit(&bars->a_empty[ai]);
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
    }
  } else {
    // Epilogue: warpgroup q = (t, h) reads columns h*64.. of A tile t (query
    // rows t*128 ..); warp w reads TMEM lanes 32*(w%4)..
    const int q = (warp - 2) >> 2;
    const int t = q & 1, h = q >> 1;
    const int quad = warp & 3;
    const int row = t * 128 + quad * 32 + lane;         // row of the 256-row query pair
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const float c2 = plan.scale2;
    int ci = 0;
    uint32_t cph = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
      const Unit1 w = decode_unit1(plan, u);
      const SeqPlan &sp = plan.seq[w.s];
      const int t_end = sp.t0 + sp.len;
      const bool active = t < w.ntiles;
      float m = -INFINITY, sum = 0.f;
      // modality of this lane's 2 keys of a block, prefetched one block ahead
      uint8_t mod_next[2];
#pragma unroll
      for (int c = 0; c < 2; ++c) {
        const int key = sp.t0 + w.b0 * kKeysPerBlock1 + h * 64 + c * 32 + lane;
        mod_next[c] = (active && key < t_end) ? modality[key] : 0;
      }
      // causal rows: this lane's row (token r of the query span) sees keys up to len - n_q + r
      const int see = sp.len - sp.n_q + (w.qp * 256 + row) / G;
      for (int b = w.b0; b < w.b1; ++b) {
        uint32_t mask[2], rmask[2];   // keys of the chunk (warp-uniform); and those this lane's row sees
        const int key_base = sp.t0 + b * kKeysPerBlock1 + h * 64;
#pragma unroll
        for (int c = 0; c < 2; ++c) {
          const int key = key_base + c * 32 + lane;
          mask[c] = __ballot_sync(0xffffffffu, key < t_end && (CAUSAL || is_mm(mod_next[c])));
          rmask[c] = mask[c];
          if (CAUSAL) {        // keys at local index <= see
            const int lim = see - (key_base - sp.t0 + c * 32);
            rmask[c] &= lim >= 31 ? 0xffffffffu : (lim < 0 ? 0u : (2u << lim) - 1u);
          }
        }
        if (active && b + 1 < w.b1) {
#pragma unroll
          for (int c = 0; c < 2; ++c) {
            const int key = key_base + kKeysPerBlock1 + c * 32 + lane;
            mod_next[c] = key < t_end ? modality[key] : 0;
          }
        }
        if (!wait_or_abort(&bars->acc_full[ci], cph, bars, err, 16)) { ok = false; break; }
        tc_fence_after();
        if (active && (mask[0] | mask[1])) {
          const uint32_t tcol = bars->tmem_base + lane_off + ci * 256 + t * 128 + h * 64;
          uint32_t rr[64];
          tmem_ld64_wait(tcol, rr);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[ci]);   // registers hold the data: release early
          online_chunk<0>(rr, rmask[0], c2, m, sum);
          online_chunk<32>(rr, rmask[1], c2, m, sum);
        } else {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[ci]);
        }
        if (++ci == 2) { ci = 0; cph ^= 1; }
      }
      if (!ok) break;
      // each column half is its own split partial; the merge combines them in a fixed order
      const int rho = w.qp * 256 + row;                  // linear row of the head group
      if (active && rho < G * sp.n_q) {
        const int r = rho / G, j = rho - r * G;
        part[(static_cast<size_t>(2 * w.split + h) * plan.total_qrows + sp.q_off + r) * plan.hq + w.g * G + j] =
            make_float2(m, sum);
      }
    }
  }
  finish_common(bars, warp, warp == 1 && lane == 0);
}

// ------------------------------------------------------------------ repack
// Packed Q: for each sequence and KV head group g, rows rho = token * G + j hold
// query head g*G + j of that token (16-byte vectors, zero padding to 256 rows).
__global__ void q_pack_kernel(const __grid_constant__ ScorePlan plan, const uint4 *__restrict__ q,
                              uint4 *__restrict__ qp, int64_t row_begin, int64_t n_vec) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n_vec) return;
  const int64_t prow = row_begin + e / 16;
  const int v = static_cast<int>(e % 16);
  int s = 0;
  while (s + 1 < plan.nseq && plan.seq[s + 1].qp_base <= prow) ++s;
  const SeqPlan &sp = plan.seq[s];
  const int local = static_cast<int>(prow - sp.qp_base);
  const int g = local / sp.rows_pad, rho = local - g * sp.rows_pad;
  const int G = plan.group;
  uint4 val = make_uint4(0, 0, 0, 0);
  if (rho < G * sp.n_q) {
    const int r = rho / G, j = rho - r * G;
    val = q[(static_cast<int64_t>(sp.q_off + r) * plan.hq + g * G + j) * 16 + v];
  }
  qp[prow * 16 + v] = val;
}

// ------------------------------------------------------------------ merge
// One thread per normaliser entry (sequence, KV head, 128-row chunk, column);
// writes -lse2 (padding columns -inf, so that they add exp2(-inf) = 0).
__global__ void lse_merge_kernel(const __grid_constant__ ScorePlan plan, const float2 *__restrict__ part,
                                 float *__restrict__ nlse2, int64_t n_entries, int64_t entry_base) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n_entries) return;
  const int64_t chunk = entry_base / kBRows + e / kBRows;
  const int col = static_cast<int>(e % kBRows);
  int s = 0;
  while (s + 1 < plan.nseq && plan.seq[s + 1].chunk_base <= chunk) ++s;
  const SeqPlan &sp = plan.seq[s];
  const int G = plan.group;
  const int nch = n_chunks(sp, G);
  const int local = static_cast<int>(chunk - sp.chunk_base);
  const int g = local / nch, c = local - g * nch;
  const int rho = c * kBRows + col;
  float out = -INFINITY;
  if (rho < G * sp.n_q) {
    const int r = rho / G, j = rho - r * G;
    const int qrow = sp.q_off + r;
    const int h = g * G + j;
    const int np = 2 * sp.n_split;   // two column halves per split
    float mm = -INFINITY;
    for (int p = 0; p < np; ++p)
      mm = fmaxf(mm, part[(static_cast<size_t>(p) * plan.total_qrows + qrow) * plan.hq + h].x);
    if (mm == -INFINITY) {
      out = INFINITY;   // no key at all (S empty): no score is written for this sequence
    } else {
      float tot = 0.f;
      for (int p = 0; p < np; ++p) {
        const float2 v = part[(static_cast<size_t>(p) * plan.total_qrows + qrow) * plan.hq + h];
        if (v.x != -INFINITY) tot += v.y * exp2f(v.x - mm);
      }
      out = -(mm + log2f(tot));
    }
  }
  nlse2[chunk * kBRows + col] = out;
}

// ------------------------------------------------------------------ pass 2
struct Unit2 {
  int s, kp, g, ntiles;
};

__device__ __forceinline__ Unit2 decode_unit2(const ScorePlan &p, int u) {
  Unit2 w;
  w.s = find_seq(p, u);
  const int local = u - p.seq[w.s].unit_begin;
  w.g = local % p.hkv;
  w.kp = local / p.hkv;
  const int keys = min(kKeysPerUnit2, p.seq[w.s].len - w.kp * kKeysPerUnit2);
  w.ntiles = keys > 128 ? 2 : 1;
  return w;
}

// a[0..3] += 2^(x c2 + nl[col]) over 32 columns (four independent partial sums).
template <int OFF>
__device__ __forceinline__ void colsum_chunk(const uint32_t (&r)[64], const float *nl, float c2, float2 (&a)[4]) {
  const float2 cc = make_float2(c2, c2);
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 L = *reinterpret_cast<const float4 *>(nl + i);
    const float2 y0 = ffma2(make_float2(__uint_as_float(r[OFF + i]), __uint_as_float(r[OFF + i + 1])), cc,
                            make_float2(L.x, L.y));
    const float2 y1 = ffma2(make_float2(__uint_as_float(r[OFF + i + 2]), __uint_as_float(r[OFF + i + 3])), cc,
                            make_float2(L.z, L.w));
    a[(i >> 2) & 3] = fadd2(a[(i >> 2) & 3], make_float2(ex2_approx(y0.x), ex2_approx(y0.y)));
    a[(i >> 2) & 3] = fadd2(a[(i >> 2) & 3], make_float2(ex2_approx(y1.x), ex2_approx(y1.y)));
  }
}

// The same over the columns OFF + i >= first only (causal rows that cannot see the key drop out;
// taken only by keys inside the query span).
template <int OFF>
__device__ __forceinline__ void colsum_chunk_from(const uint32_t (&r)[64], const float *nl, float c2, int first,
                                                  float2 (&a)[4]) {
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (OFF + i >= first) a[i & 3].x += ex2_approx(fmaf(__uint_as_float(r[OFF + i]), c2, nl[i]));
}

// Work unit = (256-key pair, KV head group g); writes the group's sum for each
// key to gsum[g][key]; the final kernel adds the groups.
template <bool CAUSAL>
__global__ void __launch_bounds__(kThreads, 1)
    score_colsum_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                        const __grid_constant__ ScorePlan plan, const float *__restrict__ nlse2,
                        float *__restrict__ gsum, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t smem[];
  if (!smem_aligned(smem)) {
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 10);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  float *lse_s = reinterpret_cast<float *>(smem + kOffL);   // [3][128], indexed by B stage
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  init_common(smem, bars, warp);
  const int G = plan.group;
  constexpr uint32_t b_tx = kBBytes + kBRows * sizeof(float);

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[kBStages] = {}, apend[kAStages] = {};
      uint32_t pend_par[kBStages] = {}, apend_par[kAStages] = {};
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        const Unit2 w = decode_unit2(plan, u);
        const SeqPlan &sp = plan.seq[w.s];
        const int nch = n_chunks(sp, G);
        if (nch == 0) continue;
        if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, err, 21)) { ok = false; break; }
        uint8_t *A = smem + kOffA + ai * kABytes;
        mbar_arrive_expect_tx(&bars->a_full[ai], kABytes);
        const int key0 = sp.t0 + w.kp * kKeysPerUnit2;
        tma_load_3d(A, &kmap, &bars->a_full[ai], 0, w.g, key0);
        tma_load_3d(A + kAHalf, &kmap, &bars->a_full[ai], 64, w.g, key0);
        apend[ai] = true;
        apend_par[ai] = aph;
        for (int c = 0; c < nch; ++c) {
          if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, err, 22)) { ok = false; break; }
          // normaliser slot bi is free once the epilogue of the chunk that used it is done
          if (!wait_or_abort(&bars->l_empty[bi], bph ^ 1, bars, err, 29)) { ok = false; break; }
          uint8_t *B = smem + kOffB + bi * kBBytes;
          mbar_arrive_expect_tx(&bars->b_full[bi], b_tx);
          const int brow = sp.qp_base + w.g * sp.rows_pad + c * kBRows;
          tma_load_3d(B, &qmap, &bars->b_full[bi], 0, 0, brow);
          tma_load_3d(B + kBHalf, &qmap, &bars->b_full[bi], 64, 0, brow);
          bulk_load(lse_s + bi * kBRows, nlse2 + (static_cast<int64_t>(sp.chunk_base) + w.g * nch + c) * kBRows,
                    kBRows * sizeof(float), &bars->b_full[bi]);
          pend[bi] = true;
          pend_par[bi] = bph;
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
        }
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
      if (!ok) {
        drain_loads(bars->b_full, pend, pend_par, kBStages);
        drain_loads(bars->a_full, apend, apend_par, kAStages);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
        const Unit2 w = decode_unit2(plan, u);
        const int nch = n_chunks(plan.seq[w.s], G);
        if (nch == 0) continue;
        if (!wait_or_abort(&bars->a_full[ai], aph, bars, err, 23)) { ok = false; break; }
        const uint32_t a_base = smem_u32(smem + kOffA + ai * kABytes);
        for (int c = 0; c < nch; ++c) {
          if (!wait_or_abort(&bars->b_full[bi], bph, bars, err, 24)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, err, 25)) { ok = false; break; }
          tc_fence_after();
          issue_mma_pair(tmem, ci, a_base, smem_u32(smem + kOffB + bi * kBBytes), w.ntiles);
          tc_commit(&bars->b_empty[bi]);
          tc_commit(&bars->acc_full[ci]);
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
        if (!ok) break;
        tc_commit(&bars->a_empty[ai]);
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
    }
  } else {
    // Epilogue: warpgroup q = (t, h) reads columns h*64.. of key tile t; one key per thread.
    const int q = (warp - 2) >> 2;
    const int t = q & 1, h = q >> 1;
    const int quad = warp & 3;
    const int tkey = quad * 32 + lane;
    const int klane = t * 128 + tkey;
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const float c2 = plan.scale2;
    float *comb = reinterpret_cast<float *>(smem + kOffC) + t * 128;
    int ci = 0, li = 0;
    uint32_t cph = 0, xph = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < plan.total_units; u += gridDim.x) {
      const Unit2 w = decode_unit2(plan, u);
      const SeqPlan &sp = plan.seq[w.s];
      const int nch = n_chunks(sp, G);
      if (nch == 0) continue;
      const bool active = t < w.ntiles;
      float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
      // causal rows: only packed rows rho >= rho_min (tokens r >= key - (len - n_q)) see this key
      const int rho_min = CAUSAL ? max(0, w.kp * kKeysPerUnit2 + klane - (sp.len - sp.n_q)) * G : 0;
      for (int c = 0; c < nch; ++c) {
        if (!wait_or_abort(&bars->acc_full[ci], cph, bars, err, 26)) { ok = false; break; }
        tc_fence_after();
        if (active) {
          const float *nl = lse_s + li * kBRows + h * 64;
          const uint32_t tcol = bars->tmem_base + lane_off + ci * 256 + t * 128 + h * 64;
          uint32_t rr[64];
          tmem_ld64_wait(tcol, rr);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->acc_empty[ci]);   // registers hold the data: release early
          const int first = rho_min - (c * kBRows + h * 64);
          if (!CAUSAL || first <= 0) {
            colsum_chunk<0>(rr, nl, c2, a);
            colsum_chunk<32>(rr, nl + 32, c2, a);
          } else if (first < 64) {
            colsum_chunk_from<0>(rr, nl, c2, first, a);
            colsum_chunk_from<32>(rr, nl + 32, c2, first, a);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->l_empty[li]);
        } else {
          tc_fence_before();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&bars->acc_empty[ci]);
            mbar_arrive(&bars->l_empty[li]);
          }
        }
        if (++ci == 2) { ci = 0; cph ^= 1; }
        if (++li == kBStages) li = 0;
      }
      if (!ok) break;
      if (!active) continue;
      const float2 s01 = fadd2(a[0], a[1]), s23 = fadd2(a[2], a[3]);
      const float2 s4 = fadd2(s01, s23);
      const float mine = s4.x + s4.y;
      if (h == 1) {
        if (!wait_or_abort(&bars->comb_empty[t], xph ^ 1, bars, err, 27)) break;
        comb[tkey] = mine;
        mbar_arrive(&bars->comb_full[t]);
      } else {
        if (!wait_or_abort(&bars->comb_full[t], xph, bars, err, 28)) break;
        const float other = comb[tkey];
        mbar_arrive(&bars->comb_empty[t]);
        const int key = sp.t0 + w.kp * kKeysPerUnit2 + klane;
        if (key < sp.t0 + sp.len) gsum[static_cast<int64_t>(w.g) * plan.total_tokens + key] = mine + other;
      }
      xph ^= 1;
    }
  }
  finish_common(bars, warp, warp == 1 && lane == 0);
}

// ------------------------------------------------------------------ final
// I_i = (sum over KV head groups, in order) / (Hq n_q) for tokens of S, 0 otherwise.
__global__ void score_finalize_kernel(const __grid_constant__ ScorePlan plan, const uint8_t *__restrict__ modality,
                                      const float *__restrict__ gsum, float *__restrict__ scores, int64_t t_begin,
                                      int64_t n) {
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n) return;
  const int64_t i = t_begin + e;
  int s = 0;
  while (s + 1 < plan.nseq && plan.seq[s + 1].t0 <= i) ++s;
  const SeqPlan &sp = plan.seq[s];
  float out = 0.f;
  if (sp.n_q > 0 && is_mm(modality[i])) {
    float acc = 0.f;
    for (int g = 0; g < plan.hkv; ++g) acc += gsum[static_cast<int64_t>(g) * plan.total_tokens + i];
    out = acc / static_cast<float>(plan.hq * sp.n_q);
  }
  scores[i] = out;
}

// ------------------------------------------------------------------ host side
using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  // looked up once, by a thread-safe static initialiser (the entry point is the same on every device)
  static const EncodeTiledFn fn = [] {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<EncodeTiledFn>(p);
    return static_cast<EncodeTiledFn>(nullptr);
  }();
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

std::atomic<uint64_t> g_attr_done{0};

}  // namespace

bool make_kv_tile_map(CUtensorMap *map, const void *k, int hkv, int64_t tokens, int64_t token_stride,
                      uint32_t box_tokens) {
  return make_map(map, k, static_cast<uint64_t>(hkv), static_cast<uint64_t>(tokens), 256,
                  static_cast<uint64_t>(token_stride), 1, box_tokens);
}

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
  if (hkv > 256) return APACK_EUNSUPPORTED;
  if (T == 0) return APACK_OK;
  // few query rows per head group (e.g. the last query token only): K-read-bound CUDA-core path
  if (narrow_score_applies(seqs)) return run_score_narrow(seqs, q, k, k_token_stride, scores, ws, stream);
  const WsLayout L = workspace_layout(seqs);
  uint8_t *wsb = static_cast<uint8_t *>(ws);
  DeviceError *err = reinterpret_cast<DeviceError *>(wsb + L.err_off);
  float2 *part = reinterpret_cast<float2 *>(wsb + L.part_off);
  float *nlse2 = reinterpret_cast<float *>(wsb + L.lse_off);
  uint8_t *qp = wsb + L.qp_off;
  float *gsum = reinterpret_cast<float *>(wsb + L.gsum_off);

  if (once_per_device(g_attr_done, [] {
        cudaError_t e = cudaFuncSetAttribute(score_rowstats_kernel<false>,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
        if (e == cudaSuccess)
          e = cudaFuncSetAttribute(score_rowstats_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemBytes);
        if (e == cudaSuccess)
          e = cudaFuncSetAttribute(score_colsum_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemBytes);
        if (e == cudaSuccess)
          e = cudaFuncSetAttribute(score_colsum_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemBytes);
        return e;
      }) != cudaSuccess)
    return APACK_ECUDA;
  CUtensorMap qmap1, kmap1, qmap2, kmap2;
  const uint64_t qp_rows = static_cast<uint64_t>(L.qp_rows > 0 ? L.qp_rows : 256);
  // pass 1: A = 256-row pairs of packed Q, B = 128-key blocks; pass 2: A = 256 keys, B = 128-row chunks
  if (!make_map(&qmap1, qp, 1, qp_rows, 256, 256, 1, 256) ||
      !make_map(&kmap1, k, hkv, T, 256, k_token_stride, 1, kKeysPerBlock1) ||
      !make_map(&qmap2, qp, 1, qp_rows, 256, 256, 1, kBRows) ||
      !make_map(&kmap2, k, hkv, T, 256, k_token_stride, 1, kKeysPerUnit2))
    return APACK_ECUDA;

  const int sms = device_sm_count();
  int64_t chunk_base = 0, qp_base = 0;
  for (int s0 = 0; s0 < B; s0 += kSeqsPerLaunch) {
    const int ns = (B - s0 < kSeqsPerLaunch) ? (B - s0) : kSeqsPerLaunch;
    ScorePlan P{};
    P.nseq = ns;
    P.hq = hq;
    P.hkv = hkv;
    P.group = G;
    P.total_qrows = static_cast<int32_t>(NQ);
    P.total_tokens = static_cast<int32_t>(T);
    P.scale2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(APACK_HEAD_DIM)));
    P.causal = seqs->softmax_domain == APACK_SOFTMAX_CAUSAL_ROW;
    int64_t chunks = 0, qrows = 0, work = 0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      SeqPlan &sp = P.seq[i];
      sp.t0 = seqs->cu_seqlens_h[b];
      sp.len = seqs->cu_seqlens_h[b + 1] - sp.t0;
      sp.q_off = seqs->cu_qlens_h[b];
      sp.n_q = seqs->cu_qlens_h[b + 1] - sp.q_off;
      sp.rows_pad = ((G * sp.n_q + 255) / 256) * 256;
      sp.qp_base = static_cast<int32_t>(qp_base + qrows);
      qrows += static_cast<int64_t>(hkv) * sp.rows_pad;
      sp.chunk_base = static_cast<int32_t>(chunk_base + chunks);
      chunks += static_cast<int64_t>(hkv) * n_chunks(sp, G);
      work += static_cast<int64_t>((sp.len + kKeysPerBlock1 - 1) / kKeysPerBlock1) * hkv * n_pairs(sp);
    }
    // Pass 1 units: (split, head group, query pair); splits sized for a few units per SM.
    const int64_t target_units = 4LL * sms;
    int64_t bps_all = (work + target_units - 1) / target_units;
    if (bps_all < 4) bps_all = 4;
    int units1 = 0, units2 = 0;
    for (int i = 0; i < ns; ++i) {
      SeqPlan &sp = P.seq[i];
      const int nb = (sp.len + kKeysPerBlock1 - 1) / kKeysPerBlock1;
      int bps = static_cast<int>(bps_all);
      if ((nb + bps - 1) / bps > kMaxSplits / 2) bps = (nb + kMaxSplits / 2 - 1) / (kMaxSplits / 2);
      sp.bps = bps > 0 ? bps : 1;
      sp.n_split = (sp.n_q > 0 && nb > 0) ? (nb + sp.bps - 1) / sp.bps : 0;
      sp.unit_begin = units1;
      units1 += sp.n_split * hkv * n_pairs(sp);
    }
    // repack the query rows of this launch's sequences
    if (qrows > 0) {
      const int64_t n_vec = qrows * 16;
      q_pack_kernel<<<static_cast<unsigned>((n_vec + 255) / 256), 256, 0, stream>>>(
          P, static_cast<const uint4 *>(q), reinterpret_cast<uint4 *>(qp), qp_base, n_vec);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    P.total_units = units1;
    if (units1 > 0) {
      const int grid = units1 < sms ? units1 : sms;
      if (P.causal)
        score_rowstats_kernel<true><<<grid, kThreads, kSmemBytes, stream>>>(qmap1, kmap1, P, seqs->modality, part, err);
      else
        score_rowstats_kernel<false><<<grid, kThreads, kSmemBytes, stream>>>(qmap1, kmap1, P, seqs->modality, part, err);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    if (chunks > 0) {
      const int64_t n_entries = chunks * kBRows;
      lse_merge_kernel<<<static_cast<unsigned>((n_entries + 255) / 256), 256, 0, stream>>>(P, part, nlse2, n_entries,
                                                                                          chunk_base * kBRows);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    // Pass 2 units: (256-key pair, head group).
    for (int i = 0; i < ns; ++i) {
      P.seq[i].unit_begin = units2;
      units2 += n_keypairs(P.seq[i]) * hkv;
    }
    P.total_units = units2;
    if (units2 > 0) {
      const int grid = units2 < sms ? units2 : sms;
      if (P.causal)
        score_colsum_kernel<true><<<grid, kThreads, kSmemBytes, stream>>>(qmap2, kmap2, P, nlse2, gsum, err);
      else
        score_colsum_kernel<false><<<grid, kThreads, kSmemBytes, stream>>>(qmap2, kmap2, P, nlse2, gsum, err);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    const int64_t t_begin = P.seq[0].t0;
    const int64_t n_tok = static_cast<int64_t>(P.seq[ns - 1].t0) + P.seq[ns - 1].len - t_begin;
    if (n_tok > 0) {
      score_finalize_kernel<<<static_cast<unsigned>((n_tok + 255) / 256), 256, 0, stream>>>(P, seqs->modality, gsum,
                                                                                            scores, t_begin, n_tok);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
    chunk_base += chunks;
    qp_base += qrows;
  }
  return APACK_OK;
}

}  // namespace apack
