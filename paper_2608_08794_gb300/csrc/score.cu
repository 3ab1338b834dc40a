// score.cu -- relevance scores of Eq. inner_score (Sec. 3.2) on the tcgen05 tensor cores.
//
// I_i = 1/(Hq n_q) sum_h sum_r softmax_{j in S}(q_{r,h} . k_{j,g(h)} / sqrt(D))_i
//
// The softmax normaliser of every (query row, head) needs all keys of S before
// any per-key average can be formed, so the scores take two passes over K:
//
//  pass 1 (row statistics): D[row][key] = Q . K^T with query rows in TMEM lanes;
//     each epilogue thread owns one row and keeps an online (reference, sum of
//     exp2) over its keys.  The (row group, key block) space is cut into equal
//     contiguous ranges, one per CTA pair; a pair writes one partial (m, sum) per
//     row for each row group its range touches.
//  merge: per packed query row, the partials combine into a log2-domain
//     normaliser lse2 = log2 sum_j 2^(x_j log2(e)/sqrt(D)), stored negated (a row whose
//     logits overflowed its run's reference is recomputed there exactly).
//  pass 2 (column sums): D[key][row] = K . Q^T with keys in TMEM lanes; each
//     thread owns one key and sums 2^(x c - lse2[row]) over the rows of one KV
//     head group; a final pass adds the Hkv group sums in a fixed order and
//     scales by 1/(Hq n_q).  No atomics anywhere: scores are deterministic.
//
// Query rows are first repacked per KV head g into linear rows rho = token * G + j
// (query head g*G + j), padded to a multiple of 256, so that tiles hold no holes.
//
// Both passes run on CTA pairs (clusters of two CTAs on two SMs) with
// tcgen05.mma.cta_group::2: one M=256 x N=256 x K=16 instruction per step, issued
// by the even CTA, reads 128 rows of A and 128 rows of B from each CTA's shared
// memory and leaves each CTA's 128 rows of D (256 fp32 columns) in its own TMEM.
// Per SM that moves 64 B of operands from shared memory per clock at the full MMA
// rate, against 128 B for an M=128 x N=128 instruction on one SM, which is what
// bounded the single-CTA version.  Each CTA loads its halves of the operands with
// TMA; the copies of both CTAs complete on the even CTA's barriers
// (cp.async.bulk.tensor ... .cta_group::2), the MMA completions arrive on both CTAs'
// barriers (tcgen05.commit ... .multicast::cluster).  The stationary operand A
// (query rows in pass 1, keys in pass 2) is held for a run of streamed B tiles (key
// blocks in pass 1, query chunks in pass 2), four B stages deep; two 256-column
// accumulators alternate in TMEM.  Warp 0 issues TMA, warp 1 owns TMEM (and on the
// even CTA issues the MMAs), warps 2..17 are four epilogue warpgroups; warpgroups 2b
// and 2b + 1 read the tiles of accumulator b, 128 columns each for the CTA's 128 lanes,
// in two TMEM loads of 64.  Pass 1 takes each key block's masks (which keys count)
// from a bit array that the query repack kernel writes once per call.  Operands sit in
// 128-byte swizzled shared memory.  Persistent pairs, one CTA per SM.
#include <cmath>
#include <cstdio>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kEpiWG = 4;                         // epilogue warpgroups
constexpr int kEpiWarps = 4 * kEpiWG;
// Warpgroups 2b and 2b + 1 own accumulator buffer b (the tiles of one parity): each reads half of
// the buffer's 256 columns, in two loads of kCols, so that one pair computes while the other waits
// for its next tile.
constexpr int kPairWarps = kEpiWarps / 2;        // epilogue warps that read one buffer
constexpr int kSpan = 128;                       // columns of a tile per warpgroup of the owning pair
constexpr int kCols = 64;                        // columns per TMEM load, pass 1
constexpr int kCols2 = 32;                       // columns per TMEM load, pass 2
static_assert(2 * kSpan == 256 && 2 * kCols == kSpan && 4 * kCols2 == kSpan,
              "two warpgroups x (two or four) loads cover a 256-column tile");
// warp 0: TMA, warp 1: TMEM (+ MMA on the even CTA), then the epilogue warps, then (pass 1) the
// key-mask warp.  Nineteen warps take the same registers per thread as eighteen.
constexpr int kThreads = 32 * (2 + kEpiWarps);
constexpr uint32_t kTmemCols = 512;    // 2 accumulators x 256 fp32 columns
constexpr int kAStages = 2, kBStages = 4;
constexpr uint32_t kRows = 128;                // rows of A and of B per CTA (M/2, N/2 of the pair)
constexpr uint32_t kTileBytes = kRows * 256;   // 128 rows x 128 bf16
constexpr uint32_t kHalf = kRows * 128;        // second 64-element K half of a tile
constexpr uint32_t kIdesc = idesc_bf16_f32(256, 256);
constexpr int kBlock = 256;                    // keys per key block (pass 1) / per key unit (pass 2)
constexpr int kChunk = 256;                    // query rows per chunk (pass 2) / per row pair (pass 1)
constexpr int kPairSlots = kMaxSplits;         // pair ranges per row group (one partial each)

struct SeqPlan {
  int32_t t0, len;        // token range of the sequence in the packed batch
  int32_t q_off, n_q;     // query tokens in packed Q
  int32_t qp_base;        // first packed row of head group 0; group g starts at qp_base + g * rows_pad
  int32_t rows_pad;       // G * n_q rounded up to a multiple of 256
  int32_t nb;             // key blocks (256 keys) of the sequence
  int32_t q_pos;          // causal rows: position of query row 0 within the sequence
  int32_t unit_begin;     // pass 2: first work unit of this sequence in the launch
  int32_t flat0;          // pass 1: first flat (row group, key block) index of the sequence
  int32_t blk0;           // pass 1: first key block of the sequence in the launch's mask array
};

struct ScorePlan {
  int32_t nseq;
  int32_t total_units;     // pass 2
  int32_t pairs;           // pass 1: CTA pairs of the launch
  int32_t flat_total;      // pass 1: (row group, key block) items of the launch (< 2^31, checked)
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
  uint64_t l_full[kBStages], l_empty[kBStages];   // pass 2: normaliser slot loaded / released (this CTA)
  uint64_t comb_full[2], comb_empty[2];           // column ranges 1.. -> range 0 hand-off
  uint32_t tmem_base;
  volatile int32_t abort;
};

// Shared memory: [A x2][B x4][-lse2 x4 (pass 2)][combine 2 x (kEpiWG - 1) x 128 float2][Bars].
// The dynamic shared window is declared 1024-byte aligned (the 128-byte swizzle
// atoms of the operand tiles need it); the kernels verify it before any use.
constexpr uint32_t kOffA = 0;
constexpr uint32_t kOffB = kAStages * kTileBytes;
constexpr uint32_t kOffL = kOffB + kBStages * kTileBytes;
constexpr uint32_t kOffC = kOffL + kBStages * kChunk * sizeof(float);
constexpr uint32_t kOffBars = kOffC + 2 * (kEpiWG - 1) * kRows * sizeof(float2);
constexpr uint32_t kSmemBytes = kOffBars + 512;
static_assert(sizeof(Bars) <= 512, "barrier block");
static_assert(kSmemBytes <= 232448, "shared memory budget");

__device__ __forceinline__ bool is_mm(uint8_t m) { return m == APACK_MOD_AUDIO || m == APACK_MOD_VISUAL; }

__host__ __device__ __forceinline__ int n_pairs(const SeqPlan &sp) { return sp.rows_pad / kChunk; }
__host__ __device__ __forceinline__ int64_t pass1_items(const SeqPlan &sp, int hkv) {
  return static_cast<int64_t>(sp.nb) * hkv * n_pairs(sp);
}

// Pass 1: pair p of P owns the flat items [start(p), start(p + 1)), start(p) = p W / P,
// and the pair holding item x is ((x + 1) P - 1) / W (64-bit products of 32-bit indices).
__host__ __device__ __forceinline__ int32_t range_start(int64_t p, int64_t P, int64_t W) {
  return static_cast<int32_t>(p * W / P);
}
__host__ __device__ __forceinline__ int32_t pair_of(int64_t x, int64_t P, int64_t W) {
  return static_cast<int32_t>(((x + 1) * P - 1) / W);
}

// ---------------------------------------------------------------- cluster-pair helpers
// Barrier waits and arrivals keep the default (CTA-scope) semantics: what crosses the pair
// through them is ordered by the asynchronous proxies themselves (TMA byte counts, MMA
// commits) and by the tcgen05 fences around TMEM reads, not by generic memory accesses.
// (Cluster-scope acquire and release here made every wait and arrival a memory barrier:
// measured 1.5x slower, with memory-barrier stalls the largest stall reason.)

// Remote (or local) arrive on a barrier given by its shared::cluster address.
__device__ __forceinline__ void arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

__device__ __forceinline__ void st_cluster_u32(uint32_t cluster_addr, uint32_t v) {
  asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr), "r"(v) : "memory");
}

// 3-D tiled load into this CTA's shared memory, completion counted on a barrier of
// either CTA of the pair (given as a shared::cluster address).
__device__ __forceinline__ void tma_load_3d_pair(void *dst, const CUtensorMap *map, uint32_t bar_cluster, int32_t c0,
                                                 int32_t c1, int32_t c2) {
  asm volatile(
      "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%3, %4, "
      "%5}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1), "r"(c2)
      : "memory");
}

__device__ __forceinline__ void mma_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(kIdesc), "r"(accumulate)
      : "memory");
}

// Arrive on the barrier at this offset in both CTAs once the issued MMAs complete.
__device__ __forceinline__ void commit_pair(uint64_t *bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          smem_u32(bar)),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

// Arrive on this CTA's own barrier once the issued MMAs complete.
__device__ __forceinline__ void commit_pair_self(uint64_t *bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t *dst_smem, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst_smem)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}

struct PairCtx {
  uint32_t rank;          // 0: the even CTA (issues the MMAs), 1: its peer
  uint32_t lead_bars;     // shared::cluster address of the even CTA's Bars
  uint32_t peer_abort;    // shared::cluster address of the other CTA's abort flag
};

template <typename T>
__device__ __forceinline__ uint32_t lead_addr(const PairCtx &pc, const Bars *bars, const T *member) {
  return pc.lead_bars + static_cast<uint32_t>(reinterpret_cast<const uint8_t *>(member) -
                                              reinterpret_cast<const uint8_t *>(bars));
}

// A wait that also gives up when a role of either CTA has aborted; a timeout aborts both.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Bars *bars, const PairCtx &pc,
                                              DeviceError *err, int where) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (;;) {
    for (int i = 0; i < 32; ++i)
      if (mbar_try_wait(bar, parity)) return true;
    if (bars->abort) return false;
    if (globaltimer_ns() - t0 > kWaitLimitNs) {
      bars->abort = 1;
      st_cluster_u32(pc.peer_abort, 1u);
      raise_device_error(err, APACK_ETIMEOUT, where);
      return false;
    }
  }
}

// True when the dynamic shared window has the 1024-byte alignment the operand tiles need.
__device__ __forceinline__ bool smem_aligned(const uint8_t *smem) { return (smem_u32(smem) & 1023u) == 0; }

__device__ PairCtx init_pair(uint8_t *smem, Bars *bars, int warp) {
  PairCtx pc;
  pc.rank = cluster_ctarank();
  // Zero the operand buffers once (every tile is then fully written by its TMA boxes).
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
      mbar_init(&bars->l_full[i], 1);
      mbar_init(&bars->l_empty[i], kPairWarps);    // stage i is read by the pair owning buffer i % 2
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->acc_full[i], 1);
      mbar_init(&bars->acc_empty[i], 2 * kPairWarps);  // the owning pair's warps in both CTAs
      mbar_init(&bars->comb_full[i], (kEpiWG - 1) * 4);
      mbar_init(&bars->comb_empty[i], 4);
    }
    mbar_init(&bars->drain, 1);
    bars->abort = 0;
    fence_mbar_init();
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  pc.lead_bars = map_shared_rank(bars, 0);
  pc.peer_abort = map_shared_rank(const_cast<const int32_t *>(&bars->abort), pc.rank ^ 1u);
  cluster_sync();                      // both CTAs' barriers exist before any remote arrive or copy
  if (warp == 1) {
    tmem_alloc_pair(&bars->tmem_base, kTmemCols);
    tc_fence_before();
  }
  __syncthreads();
  tc_fence_after();
  return pc;
}

// Teardown: after an abort the MMA thread makes sure no MMA is in flight; both CTAs
// then meet (every TMEM read and every MMA of the pair is done) and free TMEM.
__device__ void finish_pair(Bars *bars, const PairCtx &pc, int warp, bool mma_thread) {
  if (mma_thread && bars->abort) {
    commit_pair_self(&bars->drain);
    mbar_wait(&bars->drain, 0, kWaitLimitNs / 4);
  }
  if (threadIdx.x == 0 && bars->abort) {
    // copies of this CTA complete on the even CTA's barriers, which this CTA cannot watch:
    // give any still in flight time to land before the pair meets (bounded)
    const uint64_t t0 = globaltimer_ns();
    while (globaltimer_ns() - t0 < 200000ull) {
    }
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();
  tc_fence_after();
  if (warp == 1) tmem_dealloc_pair(bars->tmem_base, kTmemCols);
}

// Waits (bounded, ignoring the abort flag) for TMA loads that were issued but never
// consumed, so that no copy lands in shared memory after exit (the even CTA's barriers).
__device__ void drain_loads(uint64_t *full, const bool *pending, const uint32_t *parity, int n) {
  for (int i = 0; i < n; ++i)
    if (pending[i]) mbar_wait(&full[i], parity[i], kWaitLimitNs / 4);
}

// kCols consecutive TMEM columns of this warp's 32 lanes -> registers, loaded and waited for
// in one statement (the registers are defined only once the data is there).
__device__ __forceinline__ void tmem_load_cols(uint32_t taddr, uint32_t (&r)[64]) { tmem_ld64_wait(taddr, r); }
__device__ __forceinline__ void tmem_load_cols(uint32_t taddr, uint32_t (&r)[32]) {
  tmem_ld32(taddr, r);
  tmem_wait32(r);
}

// The eight K=16 steps of one 256 x 256 x 128 product into accumulator `ci`.
__device__ __forceinline__ void issue_mma(uint32_t tmem, int ci, uint32_t a_base, uint32_t b_base) {
#pragma unroll
  for (int kk = 0; kk < 8; ++kk) {
    const uint32_t off = (kk >> 2) * kHalf + (kk & 3) * 32;
    mma_pair(tmem + ci * 256, smem_desc_sw128(a_base + off), smem_desc_sw128(b_base + off), kk > 0 ? 1u : 0u);
  }
}

// ------------------------------------------------------------------ pass 1
// A run: the part of a pair's flat range that lies in one row group (sequence s, KV head
// group g, 256-row pair qp): key blocks [b0, b1) of that row group.
struct Run {
  int s, g, qp, b0, b1;
  int x1;          // flat index after the run
  int slot;        // partial slot: pair - first pair of the row group
};

__device__ __forceinline__ int seq_of_flat(const ScorePlan &p, int x) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].flat0 <= x) ++s;
  return s;
}

__device__ __forceinline__ Run next_run(const ScorePlan &p, int x, int x_end, int pair) {
  Run r;
  r.s = seq_of_flat(p, x);
  const SeqPlan &sp = p.seq[r.s];
  const int local = x - sp.flat0;
  const int grp = local / sp.nb;                      // row group index within the sequence
  const int np = n_pairs(sp);
  r.g = grp / np;
  r.qp = grp - r.g * np;
  r.b0 = local - grp * sp.nb;
  const int grp_end = sp.flat0 + (grp + 1) * sp.nb;
  r.x1 = x_end < grp_end ? x_end : grp_end;
  r.b1 = r.b0 + (r.x1 - x);
  r.slot = pair - pair_of(sp.flat0 + grp * sp.nb, p.pairs, p.flat_total);
  return r;
}

// Online (reference, sum) update with a thread's 64 logits of a block, in log2 units.  Keys
// that do not count are first replaced by -inf (exp2 gives 0), so that one code path serves
// every mask.  The reference is the first counted block's maximum and stays fixed for the
// run: no block's sums feed back into the next block's arithmetic.  A block whose sum leaves
// the safe range (a logit more than about 2^99 above the reference, or an overflow) only sets
// `bad`; such a row's normaliser is recomputed exactly by the merge kernel.  Four independent
// partial sums keep the add chains short.
constexpr float kSumLimit = 6.338253e29f;   // 2^99

__device__ __forceinline__ void online_block(uint32_t (&r)[64], uint32_t mask0, uint32_t mask1, float c2, float &m,
                                             float &sum, bool &bad) {
  if ((mask0 & mask1) != 0xffffffffu) {
    if ((mask0 | mask1) == 0u) return;
    const uint32_t ninf = __float_as_uint(-INFINITY);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
      r[i] = ((mask0 >> i) & 1u) ? r[i] : ninf;
      r[32 + i] = ((mask1 >> i) & 1u) ? r[32 + i] : ninf;
    }
  }
  if (m == -INFINITY) {
    float mx = __uint_as_float(r[0]);
#pragma unroll
    for (int i = 1; i < 64; ++i) mx = fmaxf(mx, __uint_as_float(r[i]));
    m = mx * c2;
  }
  float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
  const float2 cc = make_float2(c2, c2), nm = make_float2(-m, -m);
#pragma unroll
  for (int i = 0; i < 64; i += 2) {
    const float2 y = ffma2(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), cc, nm);
    a[(i >> 1) & 3] = fadd2(a[(i >> 1) & 3], make_float2(ex2_approx(y.x), ex2_approx(y.y)));
  }
  const float2 s01 = fadd2(a[0], a[1]), s23 = fadd2(a[2], a[3]);
  const float2 s4 = fadd2(s01, s23);
  const float t = s4.x + s4.y;
  bad |= !(t <= kSumLimit);
  sum += t;
}

template <bool CAUSAL>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    score_rowstats_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                          const __grid_constant__ ScorePlan plan, const uint32_t *__restrict__ mask_words,
                          float2 *__restrict__ part, DeviceError *err) {
  pdl_wait_and_release();
  extern __shared__ __align__(1024) uint8_t smem[];
  if (!smem_aligned(smem)) {   // the same in both CTAs of the pair: both leave here
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 10);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const PairCtx pc = init_pair(smem, bars, warp);
  const int G = plan.group;
  const int pair = blockIdx.x >> 1;
  const int x_begin = range_start(pair, plan.pairs, plan.flat_total);
  const int x_end = range_start(pair + 1, plan.pairs, plan.flat_total);
  const int row_half = static_cast<int>(pc.rank) * kRows;   // this CTA's rows of the 256-row pair

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[kBStages] = {}, apend[kAStages] = {};
      uint32_t pend_par[kBStages] = {}, apend_par[kAStages] = {};
      bool ok = true;
      for (int x = x_begin; ok && x < x_end;) {
        const Run w = next_run(plan, x, x_end, pair);
        const SeqPlan &sp = plan.seq[w.s];
        x = w.x1;
        if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, pc, err, 11)) { ok = false; break; }
        uint8_t *A = smem + kOffA + ai * kTileBytes;
        if (pc.rank == 0) mbar_arrive_expect_tx(&bars->a_full[ai], 2 * kTileBytes);
        const uint32_t afull = lead_addr(pc, bars, &bars->a_full[ai]);
        const int arow = sp.qp_base + w.g * sp.rows_pad + w.qp * kChunk + row_half;
        tma_load_3d_pair(A, &qmap, afull, 0, 0, arow);
        tma_load_3d_pair(A + kHalf, &qmap, afull, 64, 0, arow);
        apend[ai] = true;
        apend_par[ai] = aph;
        for (int b = w.b0; b < w.b1; ++b) {
          if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, pc, err, 12)) { ok = false; break; }
          uint8_t *B = smem + kOffB + bi * kTileBytes;
          if (pc.rank == 0) mbar_arrive_expect_tx(&bars->b_full[bi], 2 * kTileBytes);
          const uint32_t bfull = lead_addr(pc, bars, &bars->b_full[bi]);
          const int key0 = sp.t0 + b * kBlock + row_half;
          tma_load_3d_pair(B, &kmap, bfull, 0, w.g, key0);
          tma_load_3d_pair(B + kHalf, &kmap, bfull, 64, w.g, key0);
          pend[bi] = true;
          pend_par[bi] = bph;
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
        }
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
      if (!ok && pc.rank == 0) {
        drain_loads(bars->b_full, pend, pend_par, kBStages);
        drain_loads(bars->a_full, apend, apend_par, kAStages);
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && pc.rank == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int x = x_begin; ok && x < x_end;) {
        const Run w = next_run(plan, x, x_end, pair);
        x = w.x1;
        if (!wait_or_abort(&bars->a_full[ai], aph, bars, pc, err, 13)) { ok = false; break; }
        const uint32_t a_base = smem_u32(smem + kOffA + ai * kTileBytes);
        for (int b = w.b0; b < w.b1; ++b) {
          if (!wait_or_abort(&bars->b_full[bi], bph, bars, pc, err, 14)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, pc, err, 15)) { ok = false; break; }
          tc_fence_after();
          issue_mma(tmem, ci, a_base, smem_u32(smem + kOffB + bi * kTileBytes));
          commit_pair(&bars->b_empty[bi]);
          commit_pair(&bars->acc_full[ci]);
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
        if (!ok) break;
        commit_pair(&bars->a_empty[ai]);
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
    }
  } else {
    // Epilogue: warpgroup q reads the blocks of accumulator buffer q / 2 (every other block), its
    // columns (q % 2) * 128.. (keys of the block) for the CTA's 128 rows; warp w reads TMEM lanes
    // 32*(w%4)..
    const int q = (warp - 2) >> 2;
    const int own = q >> 1;                                  // accumulator buffer of this warpgroup
    const int col_base = (q & 1) * kSpan;
    const int quad = warp & 3;
    const int row = row_half + quad * 32 + lane;            // row of the 256-row pair
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t acc_empty0 = lead_addr(pc, bars, &bars->acc_empty[0]);
    const float c2 = plan.scale2;
    float2 *comb = reinterpret_cast<float2 *>(smem + kOffC);   // [2 parities][kEpiWG - 1 ranges][128 rows]
    int ci = 0;
    uint32_t cph = 0, xph = 0;
    bool ok = true;
    for (int x = x_begin; ok && x < x_end;) {
      const Run w = next_run(plan, x, x_end, pair);
      const SeqPlan &sp = plan.seq[w.s];
      x = w.x1;
      float m = -INFINITY, sum = 0.f;
      bool bad = false;
      // causal rows: this lane's row (token r of the query span) sees keys up to q_pos + r
      const int see = sp.q_pos + (w.qp * kChunk + row) / G;
      // the warpgroup's four 32-key mask words of a block (which keys count), one own block
      // ahead: lane i < 4 holds word i, shuffled to every lane when the block is taken
      const uint32_t *mwords = mask_words + sp.blk0 * 8 + (q & 1) * 4 + (lane & 3);
      const int b_first = w.b0 + ((own - ci + 2) & 1);       // blocks alternate between the buffers
      uint32_t m_next = (b_first < w.b1 && lane < 4) ? __ldg(mwords + b_first * 8) : 0u;
      for (int b = w.b0; b < w.b1; ++b) {
        if (ci == own) {
          const uint32_t m_mine = m_next;
          if (b + 2 < w.b1 && lane < 4) m_next = __ldg(mwords + (b + 2) * 8);
          const uint4 mk = make_uint4(__shfl_sync(0xffffffffu, m_mine, 0), __shfl_sync(0xffffffffu, m_mine, 1),
                                      __shfl_sync(0xffffffffu, m_mine, 2), __shfl_sync(0xffffffffu, m_mine, 3));
          // the keys of this thread's words that count; and those this lane's row sees
          uint32_t rm[4] = {mk.x, mk.y, mk.z, mk.w};
          if (CAUSAL) {        // keys at local index <= see
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              const int lim = see - (b * kBlock + col_base + 32 * i);
              rm[i] &= lim >= 31 ? 0xffffffffu : (lim < 0 ? 0u : (2u << lim) - 1u);
            }
          }
          if (!wait_or_abort(&bars->acc_full[ci], cph, bars, pc, err, 16)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const bool any = (h == 0 ? (mk.x | mk.y) : (mk.z | mk.w)) != 0u;   // uniform over the warp
            uint32_t rr[kCols];
            if (any) tmem_load_cols(bars->tmem_base + lane_off + ci * 256 + col_base + h * kCols, rr);
            if (h == 1) {     // both halves are in registers: release the buffer
              tc_fence_before();
              __syncwarp();
              if (lane == 0) arrive_cluster(acc_empty0 + ci * 8);
            }
            if (any) online_block(rr, rm[2 * h], rm[2 * h + 1], c2, m, sum, bad);
          }
        }
        if (++ci == 2) { ci = 0; cph ^= 1; }
      }
      if (!ok) break;
      // the column ranges of each row combine in a fixed order (range 0 writes the pair's
      // partial of the row group; the merge combines the pairs' partials in pair order).  A
      // sum out of range travels as a negative sum: the merge then recomputes the row.
      if (bad) sum = -1.f;
      float2 *cb = comb + (xph & 1) * (kEpiWG - 1) * kRows;
      const int trow = quad * 32 + lane;
      if (q > 0) {
        if (!wait_or_abort(&bars->comb_empty[xph & 1], ((xph >> 1) & 1) ^ 1, bars, pc, err, 17)) break;
        cb[(q - 1) * kRows + trow] = make_float2(m, sum);
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->comb_full[xph & 1]);
      } else {
        if (!wait_or_abort(&bars->comb_full[xph & 1], (xph >> 1) & 1, bars, pc, err, 18)) break;
        float2 v[kEpiWG];
        v[0] = make_float2(m, sum);
#pragma unroll
        for (int i = 1; i < kEpiWG; ++i) v[i] = cb[(i - 1) * kRows + trow];
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->comb_empty[xph & 1]);
        float mm = v[0].x;
        bool flagged = v[0].y < 0.f;
#pragma unroll
        for (int i = 1; i < kEpiWG; ++i) {
          mm = fmaxf(mm, v[i].x);
          flagged |= v[i].y < 0.f;
        }
        float tot = 0.f;
        if (mm != -INFINITY) {
#pragma unroll
          for (int i = 0; i < kEpiWG; ++i)
            if (v[i].x != -INFINITY) tot += v[i].y * exp2f(v[i].x - mm);
        }
        if (flagged) tot = -1.f;
        const int rho = w.qp * kChunk + row;                  // linear row of the head group
        if (rho < G * sp.n_q) {
          const int r = rho / G, j = rho - r * G;
          part[(static_cast<size_t>(w.slot) * plan.total_qrows + sp.q_off + r) * plan.hq + w.g * G + j] =
              make_float2(mm, tot);
        }
      }
      ++xph;
    }
  }
  finish_pair(bars, pc, warp, warp == 1 && lane == 0 && pc.rank == 0);
}

// ------------------------------------------------------------------ repack
// Packed Q: for each sequence and KV head group g, rows rho = token * G + j hold
// query head g*G + j of that token (16-byte vectors, zero padding to 256 rows).
__global__ void q_pack_kernel(const __grid_constant__ ScorePlan plan, const uint4 *__restrict__ q,
                              uint4 *__restrict__ qp, int64_t row_begin, int64_t n_vec,
                              const uint8_t *__restrict__ modality, uint32_t *__restrict__ mask_words,
                              int64_t n_words) {
  pdl_wait_and_release();
  const int64_t e = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (e >= n_vec) {
    // pass 1's key masks: word c of block b of a sequence has bit k set when key 32c + k of the
    // block is in the sequence and counts in the denominator (in S; every key in the causal
    // domain, whose per-row limit the epilogue applies)
    const int64_t wd = e - n_vec;
    if (wd >= n_words) return;
    const int gb = static_cast<int>(wd >> 3), c = static_cast<int>(wd & 7);
    int s = 0;
    while (s + 1 < plan.nseq && plan.seq[s + 1].blk0 <= gb) ++s;
    const SeqPlan &sp = plan.seq[s];
    const int key0 = sp.t0 + (gb - sp.blk0) * kBlock + c * 32, t_end = sp.t0 + sp.len;
    uint32_t word = 0;
    for (int k = 0; k < 32; ++k) {
      const int key = key0 + k;
      if (key < t_end && (plan.causal || is_mm(modality[key]))) word |= 1u << k;
    }
    mask_words[wd] = word;
    return;
  }
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
// One warp per packed query row (sequence, KV head group, rho); writes -lse2 at the row's
// packed index (padding rows -inf, so that they add exp2(-inf) = 0).  Lane p takes the partial
// of pair range p (at most 32), and a fixed shuffle tree combines them: deterministic.
//
// A row with a partial marked out of range (negative sum: a logit far above its run's
// reference) is recomputed exactly here instead: the warp's lanes take every 32nd key of
// the sequence, dot it with the row's query vector in fp32 from the bf16 values, keep an
// online (max, sum of exp2) with exact rescaling, and combine in a fixed order.  Slow, and
// only taken for inputs whose logits span more than about 99 binary orders of magnitude.
template <bool CAUSAL>
__global__ void lse_merge_kernel(const __grid_constant__ ScorePlan plan, const float2 *__restrict__ part,
                                 const uint16_t *__restrict__ qp, const uint8_t *__restrict__ k,
                                 int64_t k_stride, const uint8_t *__restrict__ modality, float *__restrict__ nlse2,
                                 int64_t row_begin, int64_t n_rows) {
  pdl_wait_and_release();
  __shared__ float qsh[8][128];                           // the query row of each warp (fallback only)
  const int64_t e = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31, wib = threadIdx.x >> 5;
  if (e >= n_rows) return;
  const int64_t prow = row_begin + e;
  int s = 0;
  while (s + 1 < plan.nseq && plan.seq[s + 1].qp_base <= prow) ++s;
  const SeqPlan &sp = plan.seq[s];
  const int G = plan.group;
  const int local = static_cast<int>(prow - sp.qp_base);
  const int g = local / sp.rows_pad, rho = local - g * sp.rows_pad;
  if (rho >= G * sp.n_q) {
    if (lane == 0) nlse2[prow] = -INFINITY;
    return;
  }
  const int r = rho / G, j = rho - r * G;
  const int qrow = sp.q_off + r;
  const int h = g * G + j;
  // the pair ranges that touched this row group, one partial each
  const int grp = g * n_pairs(sp) + rho / kChunk;
  const int x0 = sp.flat0 + grp * sp.nb;
  const int np = sp.nb > 0 ? pair_of(x0 + sp.nb - 1, plan.pairs, plan.flat_total) -
                                 pair_of(x0, plan.pairs, plan.flat_total) + 1
                           : 0;
  float2 v = make_float2(-INFINITY, 0.f);
  if (lane < np) v = part[(static_cast<size_t>(lane) * plan.total_qrows + qrow) * plan.hq + h];
  float out;
  if (__ballot_sync(0xffffffffu, v.y < 0.f) == 0u) {
    float mm = v.x;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, o));
    float tot = (v.x != -INFINITY) ? v.y * exp2f(v.x - mm) : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    out = mm == -INFINITY ? INFINITY : -(mm + log2f(tot));   // no key at all (S empty): nothing is scored
  } else {
    float *qv = qsh[wib];
    const uint16_t *qr = qp + prow * 128;
    for (int d = lane; d < 128; d += 32) qv[d] = __uint_as_float(static_cast<uint32_t>(qr[d]) << 16);
    __syncwarp();
    const int see = sp.q_pos + r;                         // causal rows: keys up to the row's position
    float m = -INFINITY, sum = 0.f;
    for (int key = sp.t0 + lane; key < sp.t0 + sp.len; key += 32) {
      if (CAUSAL ? key - sp.t0 > see : !is_mm(modality[key])) continue;
      const uint16_t *kr = reinterpret_cast<const uint16_t *>(k + key * k_stride) + g * 128;
      float dot = 0.f;
#pragma unroll 16
      for (int d = 0; d < 128; ++d) dot = fmaf(qv[d], __uint_as_float(static_cast<uint32_t>(kr[d]) << 16), dot);
      const float y = dot * plan.scale2;
      if (y > m) {
        sum = (m == -INFINITY ? 0.f : sum * exp2f(m - y)) + 1.f;
        m = y;
      } else {
        sum += exp2f(y - m);
      }
    }
    float mm = m;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mm = fmaxf(mm, __shfl_xor_sync(0xffffffffu, mm, o));
    float tot = (m != -INFINITY) ? sum * exp2f(m - mm) : 0.f;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    out = mm == -INFINITY ? INFINITY : -(mm + log2f(tot));
  }
  if (lane == 0) nlse2[prow] = out;
}

// ------------------------------------------------------------------ pass 2
struct Unit2 {
  int s, kp, g;
};

__device__ __forceinline__ Unit2 decode_unit2(const ScorePlan &p, int u) {
  Unit2 w;
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit_begin <= u) ++s;
  w.s = s;
  const int local = u - p.seq[s].unit_begin;
  w.g = local % p.hkv;
  w.kp = local / p.hkv;
  return w;
}

// a[0..3] += 2^(x c2 + nl[col]) over the 32 columns of one load (four independent partial sums).
__device__ __forceinline__ void colsum_word(const uint32_t (&r)[kCols2], const float *nl, float c2, float2 (&a)[4]) {
  const float2 cc = make_float2(c2, c2);
#pragma unroll
  for (int i = 0; i < 32; i += 4) {
    const float4 L = *reinterpret_cast<const float4 *>(nl + i);
    const float2 y0 = ffma2(make_float2(__uint_as_float(r[i]), __uint_as_float(r[i + 1])), cc, make_float2(L.x, L.y));
    const float2 y1 =
        ffma2(make_float2(__uint_as_float(r[i + 2]), __uint_as_float(r[i + 3])), cc, make_float2(L.z, L.w));
    a[(i >> 2) & 3] = fadd2(a[(i >> 2) & 3], make_float2(ex2_approx(y0.x), ex2_approx(y0.y)));
    a[(i >> 2) & 3] = fadd2(a[(i >> 2) & 3], make_float2(ex2_approx(y1.x), ex2_approx(y1.y)));
  }
}

// The same over the columns i >= first only (causal rows that cannot see the key drop out;
// taken only by keys inside the query span).
__device__ __forceinline__ void colsum_word_from(const uint32_t (&r)[kCols2], const float *nl, float c2, int first,
                                                 float2 (&a)[4]) {
#pragma unroll
  for (int i = 0; i < 32; ++i)
    if (i >= first) a[i & 3].x += ex2_approx(fmaf(__uint_as_float(r[i]), c2, nl[i]));
}

// Work unit = (256 keys, KV head group g): 128 keys per CTA of the pair; writes the group's
// sum for each key to gsum[g][key]; the final kernel adds the groups.
template <bool CAUSAL>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    score_colsum_kernel(const __grid_constant__ CUtensorMap qmap, const __grid_constant__ CUtensorMap kmap,
                        const __grid_constant__ ScorePlan plan, const float *__restrict__ nlse2,
                        float *__restrict__ gsum, DeviceError *err) {
  pdl_wait_and_release();
  extern __shared__ __align__(1024) uint8_t smem[];
  if (!smem_aligned(smem)) {   // the same in both CTAs of the pair: both leave here
    if (threadIdx.x == 0) raise_device_error(err, APACK_EDEVICE, 10);
    return;
  }
  Bars *bars = reinterpret_cast<Bars *>(smem + kOffBars);
  float *lse_s = reinterpret_cast<float *>(smem + kOffL);   // [4][256], indexed by B stage
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const PairCtx pc = init_pair(smem, bars, warp);
  const int G = plan.group;
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const int row_half = static_cast<int>(pc.rank) * kRows;   // this CTA's keys of a unit, rows of a chunk

  if (warp == 0) {
    if (lane == 0) {
      tma_prefetch_desc(&qmap);
      tma_prefetch_desc(&kmap);
      int ai = 0, bi = 0;
      uint32_t aph = 0, bph = 0;
      bool pend[kBStages] = {}, apend[kAStages] = {};
      uint32_t pend_par[kBStages] = {}, apend_par[kAStages] = {};
      bool ok = true;
      for (int u = pair; ok && u < plan.total_units; u += npairs) {
        const Unit2 w = decode_unit2(plan, u);
        const SeqPlan &sp = plan.seq[w.s];
        const int nch = sp.rows_pad / kChunk;
        if (nch == 0) continue;
        if (!wait_or_abort(&bars->a_empty[ai], aph ^ 1, bars, pc, err, 21)) { ok = false; break; }
        uint8_t *A = smem + kOffA + ai * kTileBytes;
        if (pc.rank == 0) mbar_arrive_expect_tx(&bars->a_full[ai], 2 * kTileBytes);
        const uint32_t afull = lead_addr(pc, bars, &bars->a_full[ai]);
        const int key0 = sp.t0 + w.kp * kBlock + row_half;
        tma_load_3d_pair(A, &kmap, afull, 0, w.g, key0);
        tma_load_3d_pair(A + kHalf, &kmap, afull, 64, w.g, key0);
        apend[ai] = true;
        apend_par[ai] = aph;
        for (int c = 0; c < nch; ++c) {
          if (!wait_or_abort(&bars->b_empty[bi], bph ^ 1, bars, pc, err, 22)) { ok = false; break; }
          // normaliser slot bi is free once this CTA's epilogue of the chunk that used it is done
          if (!wait_or_abort(&bars->l_empty[bi], bph ^ 1, bars, pc, err, 29)) { ok = false; break; }
          const int64_t row0 = static_cast<int64_t>(sp.qp_base) + w.g * sp.rows_pad + c * kChunk;
          mbar_arrive_expect_tx(&bars->l_full[bi], kChunk * sizeof(float));
          bulk_load(lse_s + bi * kChunk, nlse2 + row0, kChunk * sizeof(float), &bars->l_full[bi]);
          uint8_t *B = smem + kOffB + bi * kTileBytes;
          if (pc.rank == 0) mbar_arrive_expect_tx(&bars->b_full[bi], 2 * kTileBytes);
          const uint32_t bfull = lead_addr(pc, bars, &bars->b_full[bi]);
          tma_load_3d_pair(B, &qmap, bfull, 0, 0, static_cast<int32_t>(row0) + row_half);
          tma_load_3d_pair(B + kHalf, &qmap, bfull, 64, 0, static_cast<int32_t>(row0) + row_half);
          pend[bi] = true;
          pend_par[bi] = bph;
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
        }
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
      if (!ok) {
        // this CTA's normaliser copies complete on its own barriers
        drain_loads(bars->l_full, pend, pend_par, kBStages);
        if (pc.rank == 0) {
          drain_loads(bars->b_full, pend, pend_par, kBStages);
          drain_loads(bars->a_full, apend, apend_par, kAStages);
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && pc.rank == 0) {
      int ai = 0, bi = 0, ci = 0;
      uint32_t aph = 0, bph = 0, cph = 0;
      const uint32_t tmem = bars->tmem_base;
      bool ok = true;
      for (int u = pair; ok && u < plan.total_units; u += npairs) {
        const Unit2 w = decode_unit2(plan, u);
        const int nch = plan.seq[w.s].rows_pad / kChunk;
        if (nch == 0) continue;
        if (!wait_or_abort(&bars->a_full[ai], aph, bars, pc, err, 23)) { ok = false; break; }
        const uint32_t a_base = smem_u32(smem + kOffA + ai * kTileBytes);
        for (int c = 0; c < nch; ++c) {
          if (!wait_or_abort(&bars->b_full[bi], bph, bars, pc, err, 24)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_empty[ci], cph ^ 1, bars, pc, err, 25)) { ok = false; break; }
          tc_fence_after();
          issue_mma(tmem, ci, a_base, smem_u32(smem + kOffB + bi * kTileBytes));
          commit_pair(&bars->b_empty[bi]);
          commit_pair(&bars->acc_full[ci]);
          if (++bi == kBStages) { bi = 0; bph ^= 1; }
          if (++ci == 2) { ci = 0; cph ^= 1; }
        }
        if (!ok) break;
        commit_pair(&bars->a_empty[ai]);
        if (++ai == kAStages) { ai = 0; aph ^= 1; }
      }
    }
  } else {
    // Epilogue: warpgroup q reads the chunks of accumulator buffer q / 2 (every other chunk), its
    // columns (q % 2) * 128.. (rows of the chunk); one key per thread.
    const int q = (warp - 2) >> 2;
    const int own = q >> 1;                                  // accumulator buffer of this warpgroup
    const int col_base = (q & 1) * kSpan;
    const int quad = warp & 3;
    const int tkey = quad * 32 + lane;
    const int klane = row_half + tkey;                  // key of the 256-key unit
    const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
    const uint32_t acc_empty0 = lead_addr(pc, bars, &bars->acc_empty[0]);
    const float c2 = plan.scale2;
    float *comb = reinterpret_cast<float *>(smem + kOffC);   // [2 parities][kEpiWG - 1 ranges][128 keys]
    int ci = 0, li = 0;
    uint32_t cph = 0, lph = 0, xph = 0;
    bool ok = true;
    for (int u = pair; ok && u < plan.total_units; u += npairs) {
      const Unit2 w = decode_unit2(plan, u);
      const SeqPlan &sp = plan.seq[w.s];
      const int nch = sp.rows_pad / kChunk;
      if (nch == 0) continue;
      float2 a[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
      // causal rows: only packed rows rho >= rho_min (tokens r >= key - q_pos) see this key
      const int rho_min = CAUSAL ? max(0, w.kp * kBlock + klane - sp.q_pos) * G : 0;
      for (int c = 0; c < nch; ++c) {
        if (ci == own) {   // chunks alternate between the buffers (normaliser slot li % 2 == ci)
          if (!wait_or_abort(&bars->l_full[li], lph, bars, pc, err, 30)) { ok = false; break; }
          if (!wait_or_abort(&bars->acc_full[ci], cph, bars, pc, err, 26)) { ok = false; break; }
          tc_fence_after();
#pragma unroll
          for (int h = 0; h < kSpan / kCols2; ++h) {
            const int col0 = col_base + h * kCols2;
            const float *nl = lse_s + li * kChunk + col0;
            uint32_t rr[kCols2];
            tmem_load_cols(bars->tmem_base + lane_off + ci * 256 + col0, rr);
            if (h == kSpan / kCols2 - 1) {     // every column is in registers: release the buffer
              tc_fence_before();
              __syncwarp();
              if (lane == 0) arrive_cluster(acc_empty0 + ci * 8);
            }
            const int first = rho_min - (c * kChunk + col0);
            if (!CAUSAL || first <= 0)
              colsum_word(rr, nl, c2, a);
            else if (first < kCols2)
              colsum_word_from(rr, nl, c2, first, a);
          }
          __syncwarp();
          if (lane == 0) mbar_arrive(&bars->l_empty[li]);
        }
        if (++ci == 2) { ci = 0; cph ^= 1; }
        if (++li == kBStages) { li = 0; lph ^= 1; }
      }
      if (!ok) break;
      const float2 s01 = fadd2(a[0], a[1]), s23 = fadd2(a[2], a[3]);
      const float2 s4 = fadd2(s01, s23);
      const float mine = s4.x + s4.y;
      float *cb = comb + (xph & 1) * (kEpiWG - 1) * kRows;
      if (q > 0) {
        if (!wait_or_abort(&bars->comb_empty[xph & 1], ((xph >> 1) & 1) ^ 1, bars, pc, err, 27)) break;
        cb[(q - 1) * kRows + tkey] = mine;
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->comb_full[xph & 1]);
      } else {
        if (!wait_or_abort(&bars->comb_full[xph & 1], (xph >> 1) & 1, bars, pc, err, 28)) break;
        float tot = mine;
#pragma unroll
        for (int i = 1; i < kEpiWG; ++i) tot += cb[(i - 1) * kRows + tkey];   // fixed order
        __syncwarp();
        if (lane == 0) mbar_arrive(&bars->comb_empty[xph & 1]);
        const int key = sp.t0 + w.kp * kBlock + klane;
        if (key < sp.t0 + sp.len) gsum[static_cast<int64_t>(w.g) * plan.total_tokens + key] = tot;
      }
      ++xph;
    }
  }
  finish_pair(bars, pc, warp, warp == 1 && lane == 0 && pc.rank == 0);
}

// ------------------------------------------------------------------ final
// I_i = (sum over KV head groups, in order) / (Hq n_q) for tokens of S, 0 otherwise.
__global__ void score_finalize_kernel(const __grid_constant__ ScorePlan plan, const uint8_t *__restrict__ modality,
                                      const float *__restrict__ gsum, float *__restrict__ scores, int64_t t_begin,
                                      int64_t n) {
  pdl_wait_and_release();
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
std::atomic<int> g_max_pairs[64];   // per device: CTA pairs that can be resident at once (0 = not probed)

// CTA pairs of the scoring kernels that fit the device at once (one CTA per SM).
int max_resident_pairs() {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
  if (dev < 64) {
    const int cached = g_max_pairs[dev].load(std::memory_order_relaxed);
    if (cached > 0) return cached;
  }
  int n = 0;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(2 * (device_sm_count() / 2), 1, 1);
  cfg.blockDim = dim3(kThreads, 1, 1);
  cfg.dynamicSmemBytes = kSmemBytes;
  // the kernels declare their cluster shape (__cluster_dims__), so the configuration leaves it out
  if (cudaOccupancyMaxActiveClusters(&n, score_colsum_kernel<false>, &cfg) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    n = device_sm_count() / 2;
  }
  if (n > device_sm_count() / 2) n = device_sm_count() / 2;
  if (n < 1) n = 1;
  if (dev < 64) g_max_pairs[dev].store(n, std::memory_order_relaxed);
  return n;
}

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
  // few query rows per head group (e.g. the last query token only): K-read-bound path
  if (narrow_score_applies(seqs)) return run_score_narrow(seqs, q, k, k_token_stride, scores, ws, stream);
  const WsLayout L = workspace_layout(seqs);
  uint8_t *wsb = static_cast<uint8_t *>(ws);
  DeviceError *err = reinterpret_cast<DeviceError *>(wsb + L.err_off);
  float2 *part = reinterpret_cast<float2 *>(wsb + L.part_off);
  float *nlse2 = reinterpret_cast<float *>(wsb + L.lse_off);
  uint8_t *qp = wsb + L.qp_off;
  float *gsum = reinterpret_cast<float *>(wsb + L.gsum_off);
  uint32_t *mask_words = reinterpret_cast<uint32_t *>(wsb + L.mask_off);

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
  CUtensorMap qmap, kmap;
  const uint64_t qp_rows = static_cast<uint64_t>(L.qp_rows > 0 ? L.qp_rows : 256);
  // every operand tile is 128 rows (of packed Q or of one KV head's keys) per CTA
  if (!make_map(&qmap, qp, 1, qp_rows, 256, 256, 1, kRows) || !make_map(&kmap, k, hkv, T, 256, k_token_stride, 1, kRows))
    return APACK_ECUDA;

  const int max_pairs = max_resident_pairs();
  int64_t qp_base = 0;
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
    int64_t qrows = 0, flat = 0, nb_max = 0;
    int units2 = 0, blocks = 0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      SeqPlan &sp = P.seq[i];
      sp.t0 = seqs->cu_seqlens_h[b];
      sp.len = seqs->cu_seqlens_h[b + 1] - sp.t0;
      sp.q_off = seqs->cu_qlens_h[b];
      sp.n_q = seqs->cu_qlens_h[b + 1] - sp.q_off;
      sp.rows_pad = ((G * sp.n_q + kChunk - 1) / kChunk) * kChunk;
      sp.qp_base = static_cast<int32_t>(qp_base + qrows);
      qrows += static_cast<int64_t>(hkv) * sp.rows_pad;
      sp.nb = sp.n_q > 0 ? (sp.len + kBlock - 1) / kBlock : 0;
      sp.q_pos = query_position(seqs, b);
      sp.flat0 = static_cast<int32_t>(flat);
      sp.blk0 = blocks;
      blocks += sp.nb;
      flat += pass1_items(sp, hkv);
      if (sp.nb > nb_max) nb_max = sp.nb;
      sp.unit_begin = units2;
      if (sp.rows_pad > 0) units2 += ((sp.len + kBlock - 1) / kBlock) * hkv;
    }
    // Pass 1: equal ranges of the flat (row group, key block) items per pair; a range must stay at
    // least ceil(nb_max / (kPairSlots - 1)) items long so that a row group meets at most kPairSlots
    // pairs (its partial slots).
    if (flat >= (int64_t{1} << 31) - 1) return APACK_EUNSUPPORTED;   // flat indices are 32-bit on the device
    P.flat_total = static_cast<int32_t>(flat);
    int64_t pairs1 = max_pairs;
    if (flat > 0) {
      const int64_t min_len = (nb_max + kPairSlots - 2) / (kPairSlots - 1);
      if (pairs1 > flat / min_len) pairs1 = flat / min_len;
      if (pairs1 < 1) pairs1 = 1;
    }
    P.pairs = static_cast<int32_t>(pairs1);
    // repack the query rows of this launch's sequences and write pass 1's key masks
    const int64_t n_words = static_cast<int64_t>(blocks) * (kBlock / 32);
    if (qrows > 0) {
      const int64_t n_vec = qrows * 16;
      if (check_cuda(launch_pdl(q_pack_kernel, dim3(static_cast<unsigned>((n_vec + n_words + 255) / 256)), dim3(256), 0,
                                stream, P, static_cast<const uint4 *>(q), reinterpret_cast<uint4 *>(qp), qp_base, n_vec,
                                seqs->modality, mask_words, n_words)) != APACK_OK)
        return APACK_ECUDA;
      count_launches(1);
    }
    if (flat > 0) {
      const unsigned grid = static_cast<unsigned>(2 * pairs1);
      const uint32_t *mw = mask_words;
      const cudaError_t e = P.causal ? launch_pdl(score_rowstats_kernel<true>, dim3(grid), dim3(kThreads), kSmemBytes,
                                                  stream, qmap, kmap, P, mw, part, err)
                                     : launch_pdl(score_rowstats_kernel<false>, dim3(grid), dim3(kThreads), kSmemBytes,
                                                  stream, qmap, kmap, P, mw, part, err);
      count_launches(1);
      if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
    }
    if (qrows > 0) {
      const unsigned blocks = static_cast<unsigned>((qrows * 32 + 255) / 256);   // one warp per packed row
      const uint16_t *qp16 = reinterpret_cast<const uint16_t *>(qp);
      const uint8_t *k8 = static_cast<const uint8_t *>(k);
      const float2 *pc = part;
      const int64_t qb = qp_base;
      const cudaError_t e =
          P.causal ? launch_pdl(lse_merge_kernel<true>, dim3(blocks), dim3(256), 0, stream, P, pc, qp16, k8,
                                k_token_stride, static_cast<const uint8_t *>(seqs->modality), nlse2, qb, qrows)
                   : launch_pdl(lse_merge_kernel<false>, dim3(blocks), dim3(256), 0, stream, P, pc, qp16, k8,
                                k_token_stride, static_cast<const uint8_t *>(seqs->modality), nlse2, qb, qrows);
      count_launches(1);
      if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
    }
    // Pass 2 units: (256 keys, head group), dealt round-robin to the pairs.
    P.total_units = units2;
    if (units2 > 0) {
      const int pairs2 = units2 < max_pairs ? units2 : max_pairs;
      const unsigned grid = static_cast<unsigned>(2 * pairs2);
      const float *nl = nlse2;
      const cudaError_t e = P.causal ? launch_pdl(score_colsum_kernel<true>, dim3(grid), dim3(kThreads), kSmemBytes,
                                                  stream, qmap, kmap, P, nl, gsum, err)
                                     : launch_pdl(score_colsum_kernel<false>, dim3(grid), dim3(kThreads), kSmemBytes,
                                                  stream, qmap, kmap, P, nl, gsum, err);
      count_launches(1);
      if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
    }
    const int64_t t_begin = P.seq[0].t0;
    const int64_t n_tok = static_cast<int64_t>(P.seq[ns - 1].t0) + P.seq[ns - 1].len - t_begin;
    if (n_tok > 0) {
      const float *gs = gsum;
      if (check_cuda(launch_pdl(score_finalize_kernel, dim3(static_cast<unsigned>((n_tok + 255) / 256)), dim3(256), 0,
                                stream, P, static_cast<const uint8_t *>(seqs->modality), gs, scores, t_begin,
                                n_tok)) != APACK_OK)
        return APACK_ECUDA;
      count_launches(1);
    }
    qp_base += qrows;
  }
  return APACK_OK;
}

}  // namespace apack
