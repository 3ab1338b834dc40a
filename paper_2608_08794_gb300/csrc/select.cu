// select.cu -- per-(sequence, modality) top-k of Eq. inner (Sec. 3.2) and the stable keep map.
//
// One thread-block cluster of CL CTAs per sequence (16 for long sequences when the
// launch's clusters still fit the GPU that way, else 8); CTA c owns a contiguous
// slice of the sequence's tokens.
//
//  1. Radix select (4 passes of 8 bits, most significant first) of the k-th
//     largest score of every segment.  Scores are >= 0, so the order of their
//     IEEE bit patterns as unsigned integers is their numeric order.  Each CTA
//     builds a shared-memory histogram of its slice; the cluster merges them
//     through distributed shared memory and every CTA derives the same digit.
//     The result per segment is a threshold bit pattern T and a quota q: keep
//     every score > T and the first q scores == T in token order (ties go to
//     the lower index).
//  2. Counts per warp run and per CTA (other tokens, > T, == T) are exchanged
//     through DSMEM so that each warp knows its output offset and how many
//     ties precede it.  Histogram atomics are aggregated per warp and bin.
//  3. Each warp walks its contiguous run of the slice in token order (ballot
//     prefix counts give the positions) and writes keep_idx (ascending), the
//     compacted modality and dst_of_src.
// A CTA's slice (scores as bit patterns and modality codes) is read from global
// memory once into shared memory when it fits (slices up to kMaxCached tokens);
// all passes then run on the shared copy.
#include <cstdio>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kThreads = 1024;
constexpr int kWarps = kThreads / 32;
static_assert(kWarps == 32, "the keep-offset scan gives one lane to each warp of a CTA");
constexpr int kMaxCached = 40960;               // tokens per CTA slice cached in shared memory (200 KB)
constexpr size_t kCacheBytes = static_cast<size_t>(kMaxCached) * 5;

struct SelSeq {
  int32_t t0, len;
  int32_t out_base, out_len;   // host-computed output offset and kept count
  int32_t n_seg[2];            // host counts per segment
  int32_t k[2];                // keep counts per segment
};

struct SelectPlan {
  int32_t nseq;
  int32_t nsegs;               // 2 per modality, 1 joint
  int32_t write_cu0;           // write new_cu_seqlens[0] = 0 (first launch of a batch)
  int32_t seq_base;            // index of seq[0] in the batch
  int32_t cache_tokens;        // slice tokens the dynamic shared memory holds (0: no cache)
  SelSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int seg_of(uint8_t m, int nsegs) {
  if (m == APACK_MOD_AUDIO) return 0;
  if (m == APACK_MOD_VISUAL) return nsegs == 1 ? 0 : 1;
  return -1;
}

// One token of the slice, from the shared-memory copy when there is one.
struct Tok {
  uint32_t bits;
  int seg;
  uint8_t mod;
  bool in;
};

__device__ __forceinline__ Tok load_tok(const float *__restrict__ scores, const uint8_t *__restrict__ modality,
                                        const uint32_t *c_bits, const uint8_t *c_mod, int lo, int i, int end,
                                        int nsegs) {
  Tok t;
  t.in = i < end;
  if (c_bits) {
    t.bits = t.in ? c_bits[i - lo] : 0u;
    t.mod = t.in ? c_mod[i - lo] : static_cast<uint8_t>(0xFF);
  } else {
    t.bits = t.in ? __float_as_uint(scores[i]) : 0u;
    t.mod = t.in ? modality[i] : static_cast<uint8_t>(0xFF);
  }
  t.seg = seg_of(t.mod, nsegs);
  return t;
}

// Adds one count per lane with bin >= 0.  When every counted lane of the warp
// has the same bin (the usual case for the high digits, where neighbouring
// scores share them) a single atomic carries the whole warp.
__device__ __forceinline__ void add_bin(uint32_t *h, int bin, int lane) {
  const uint32_t valid = __ballot_sync(0xffffffffu, bin >= 0);
  if (valid == 0u) return;
  const int first = __shfl_sync(0xffffffffu, bin, __ffs(valid) - 1);
  const uint32_t same = __ballot_sync(0xffffffffu, bin == first);
  if (same == valid) {
    if (lane == 0) atomicAdd(&h[first], static_cast<uint32_t>(__popc(valid)));
  } else if (bin >= 0) {
    atomicAdd(&h[bin], 1u);
  }
}

template <int CL>
__global__ void __cluster_dims__(CL, 1, 1) __launch_bounds__(kThreads)
    select_kernel(const __grid_constant__ SelectPlan plan, const float *__restrict__ scores,
                  const uint8_t *__restrict__ modality, int32_t *__restrict__ keep_idx,
                  uint8_t *__restrict__ modality_out, int32_t *__restrict__ dst_of_src,
                  int32_t *__restrict__ new_cu, DeviceError *err) {
  __shared__ uint32_t hist[2][2][256];
  __shared__ uint32_t tot[2][256];            // cluster-wide histogram of the current pass
  __shared__ uint32_t rcnt[CL][5];            // per-CTA counts of the cluster
  __shared__ uint32_t st_prefix[2], st_mask[2], st_krem[2], st_total[2];
  __shared__ uint32_t wcnt[kWarps][5];        // per warp chunk: other, gt0, gt1, eq0, eq1
  __shared__ uint32_t cnt[5];                 // per CTA (read by the cluster)
  __shared__ uint32_t wbase[kWarps], weqb[kWarps][2];
  extern __shared__ __align__(16) uint8_t cache_raw[];
  pdl_wait_and_release();                     // the scores are complete; the compaction may be scheduled

  const SelSeq &sq = plan.seq[blockIdx.y];
  const uint32_t crank = cluster_ctarank();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint32_t lt_mask = (1u << lane) - 1u;
  const int nsegs = plan.nsegs;
  const int chunk = (sq.len + CL - 1) / CL;
  const int lo = sq.t0 + min(sq.len, static_cast<int>(crank) * chunk);
  const int hi = sq.t0 + min(sq.len, static_cast<int>(crank + 1) * chunk);
  // each warp owns a contiguous run of the slice (a multiple of 32 tokens)
  const int cw = ((hi - lo) + kWarps * 32 - 1) / (kWarps * 32) * 32;
  const int wlo = min(hi, lo + warp * cw), whi = min(hi, wlo + cw);

  // shared copy of the slice: bits [n] then modality [n]
  const uint32_t *c_bits = nullptr;
  const uint8_t *c_mod = nullptr;
  const int n = hi - lo;
  if (n <= plan.cache_tokens) {
    uint32_t *wb = reinterpret_cast<uint32_t *>(cache_raw);
    uint8_t *wm = cache_raw + static_cast<size_t>(plan.cache_tokens) * 4;
    for (int x = tid; x < n; x += kThreads) {
      wb[x] = __float_as_uint(scores[lo + x]);
      wm[x] = modality[lo + x];
    }
    c_bits = wb;
    c_mod = wm;
  }
  for (int j = tid; j < 2 * 2 * 256; j += kThreads) (&hist[0][0][0])[j] = 0u;
  if (tid < 2) {
    st_prefix[tid] = 0u;
    st_mask[tid] = 0u;
    st_krem[tid] = static_cast<uint32_t>(tid < nsegs ? sq.k[tid] : 0);
    st_total[tid] = 0u;
  }
  __syncthreads();
  cluster_sync();   // every CTA's histograms are zero before anyone adds

  // ---- 1. radix select
  for (int d = 0; d < 4; ++d) {
    const int hb = d & 1;
    const int shift = 24 - 8 * d;
    const uint32_t p0 = st_prefix[0], p1 = st_prefix[1], m0 = st_mask[0], m1 = st_mask[1];
    // two 32-token rounds per iteration (independent chains)
    for (int b = wlo; b < whi; b += 64) {
      const Tok t0 = load_tok(scores, modality, c_bits, c_mod, lo, b + lane, whi, nsegs);
      const Tok t1 = load_tok(scores, modality, c_bits, c_mod, lo, b + 32 + lane, whi, nsegs);
      int bin0 = -1, bin1 = -1;
      if (t0.seg >= 0 && (t0.bits & (t0.seg ? m1 : m0)) == (t0.seg ? p1 : p0))
        bin0 = t0.seg * 256 + static_cast<int>((t0.bits >> shift) & 255u);
      if (t1.seg >= 0 && (t1.bits & (t1.seg ? m1 : m0)) == (t1.seg ? p1 : p0))
        bin1 = t1.seg * 256 + static_cast<int>((t1.bits >> shift) & 255u);
      add_bin(&hist[hb][0][0], bin0, lane);
      add_bin(&hist[hb][0][0], bin1, lane);
    }
    __syncthreads();
    cluster_sync();
    for (int j = tid; j < 2 * 256; j += kThreads) (&hist[hb ^ 1][0][0])[j] = 0u;
    // cluster-wide histogram: thread (seg, bin) adds the bin of every CTA, its
    // CL remote loads issued back to back
    for (int j = tid; j < nsegs * 256; j += kThreads) {
      uint32_t v[CL];
#pragma unroll
      for (int r = 0; r < CL; ++r) v[r] = ld_shared_cluster_u32(map_shared_rank(&(&hist[hb][0][0])[j], r));
      uint32_t sum = 0;
#pragma unroll
      for (int r = 0; r < CL; ++r) sum += v[r];
      (&tot[0][0])[j] = sum;
    }
    __syncthreads();
    if (warp < nsegs) {
      const int seg = warp;
      uint32_t c[8];
      uint32_t lsum = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        c[b] = tot[seg][lane * 8 + b];
        lsum += c[b];
      }
      // inclusive suffix sum over lanes (higher lanes hold higher digits)
      uint32_t suf = lsum;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t nb = __shfl_down_sync(0xffffffffu, suf, off);
        if (lane + off < 32) suf += nb;
      }
      const uint32_t above_lane = suf - lsum;
      const uint32_t total = __shfl_sync(0xffffffffu, suf, 0);
      const uint32_t k = st_krem[seg];
      const bool mine = k > 0 && above_lane < k && k <= suf;
      const uint32_t who = __ballot_sync(0xffffffffu, mine);
      uint32_t digit = 0, above = 0;
      if (mine) {
        uint32_t run = above_lane;
        for (int b = 7; b >= 0; --b) {
          if (run + c[b] >= k) {
            digit = static_cast<uint32_t>(lane * 8 + b);
            above = run;
            break;
          }
          run += c[b];
        }
      }
      if (who != 0u) {
        const int src = __ffs(who) - 1;
        digit = __shfl_sync(0xffffffffu, digit, src);
        above = __shfl_sync(0xffffffffu, above, src);
        if (lane == 0) {
          st_prefix[seg] |= digit << shift;
          st_mask[seg] |= 255u << shift;
          st_krem[seg] = k - above;
        }
      }
      if (d == 0 && lane == 0) st_total[seg] = total;
    }
    __syncthreads();
  }

  // Threshold and tie quota per segment.
  uint32_t T[2], quota[2];
#pragma unroll
  for (int s = 0; s < 2; ++s) {
    const bool none = s >= nsegs || sq.k[s] <= 0;
    T[s] = none ? 0xFFFFFFFFu : st_prefix[s];
    quota[s] = none ? 0u : st_krem[s];
  }

  // ---- 2. counts per warp run, per CTA, exchanged through the cluster
  {
    uint32_t c_other = 0, c_gt0 = 0, c_gt1 = 0, c_eq0 = 0, c_eq1 = 0;
    for (int b = wlo; b < whi; b += 32) {
      const Tok t = load_tok(scores, modality, c_bits, c_mod, lo, b + lane, whi, nsegs);
      const uint32_t tt = t.seg > 0 ? T[1] : T[0];
      c_other += __popc(__ballot_sync(0xffffffffu, t.in && t.seg < 0));
      c_gt0 += __popc(__ballot_sync(0xffffffffu, t.seg == 0 && t.bits > tt));
      c_gt1 += __popc(__ballot_sync(0xffffffffu, t.seg == 1 && t.bits > tt));
      c_eq0 += __popc(__ballot_sync(0xffffffffu, t.seg == 0 && t.bits == tt));
      c_eq1 += __popc(__ballot_sync(0xffffffffu, t.seg == 1 && t.bits == tt));
    }
    if (lane == 0) {
      wcnt[warp][0] = c_other;
      wcnt[warp][1] = c_gt0;
      wcnt[warp][2] = c_gt1;
      wcnt[warp][3] = c_eq0;
      wcnt[warp][4] = c_eq1;
    }
  }
  __syncthreads();
  if (tid < 5) {
    uint32_t v = 0;
    for (int w = 0; w < kWarps; ++w) v += wcnt[w][tid];
    cnt[tid] = v;
  }
  __syncthreads();
  cluster_sync();
  if (tid < CL * 5) rcnt[tid / 5][tid % 5] = ld_shared_cluster_u32(map_shared_rank(&cnt[tid % 5], tid / 5));
  __syncthreads();
  if (warp == 0) {
    // Token order runs over the CTAs of the cluster, then over the warps of this CTA: ties are
    // granted in that order until each segment's quota runs out.  Lane r stands for CTA r, then
    // for warp r; exclusive prefix sums over the lanes replace a walk in order.
    auto excl_scan = [&](uint32_t v) -> uint32_t {
      uint32_t x = v;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t y = __shfl_up_sync(0xffffffffu, x, off);
        if (lane >= off) x += y;
      }
      return x - v;
    };
    auto granted = [](uint32_t ties, uint32_t before, uint32_t q) -> uint32_t {
      const uint32_t avail = q > before ? q - before : 0u;
      return ties < avail ? ties : avail;
    };
    // the cluster's CTAs
    uint32_t c[5] = {0u, 0u, 0u, 0u, 0u};
    if (lane < CL) {
#pragma unroll
      for (int i = 0; i < 5; ++i) c[i] = rcnt[lane][i];
    }
    const uint32_t eqp0 = excl_scan(c[3]), eqp1 = excl_scan(c[4]);   // ties of the CTAs before
    const uint32_t kept = c[0] + c[1] + c[2] + granted(c[3], eqp0, quota[0]) + granted(c[4], eqp1, quota[1]);
    const uint32_t kept_excl = excl_scan(kept);
    const uint32_t kept_all = __shfl_sync(0xffffffffu, kept_excl + kept, 31);
    const uint32_t kept_before = __shfl_sync(0xffffffffu, kept_excl, static_cast<int>(crank));
    const uint32_t eqb0 = __shfl_sync(0xffffffffu, eqp0, static_cast<int>(crank));
    const uint32_t eqb1 = __shfl_sync(0xffffffffu, eqp1, static_cast<int>(crank));
    // this CTA's warps (kWarps == 32: one lane each)
    const uint32_t *wc = wcnt[lane];
    const uint32_t we0 = eqb0 + excl_scan(wc[3]), we1 = eqb1 + excl_scan(wc[4]);
    const uint32_t wk = wc[0] + wc[1] + wc[2] + granted(wc[3], we0, quota[0]) + granted(wc[4], we1, quota[1]);
    wbase[lane] = kept_before + excl_scan(wk);
    weqb[lane][0] = we0;
    weqb[lane][1] = we1;
    if (crank == 0 && lane == 0) {
      // Device-side consistency with the host counts.
      bool bad = kept_all != static_cast<uint32_t>(sq.out_len);
      for (int s = 0; s < nsegs; ++s)   // segment sizes seen by the first radix pass
        if (st_total[s] != static_cast<uint32_t>(sq.n_seg[s])) bad = true;
      if (bad) raise_device_error(err, APACK_EDEVICE, 31, plan.seq_base + static_cast<int>(blockIdx.y),
                                  static_cast<int32_t>(kept_all));
      if (new_cu) {
        if (plan.write_cu0 && blockIdx.y == 0) new_cu[0] = 0;
        new_cu[plan.seq_base + blockIdx.y + 1] = sq.out_base + sq.out_len;
      }
    }
  }
  __syncthreads();
  cluster_sync();   // all remote reads of cnt[] are done before any CTA may exit

  // ---- 3. ordered writes: each warp walks its run in token order
  uint32_t pos = wbase[warp];
  uint32_t er0 = weqb[warp][0], er1 = weqb[warp][1];
  for (int b = wlo; b < whi; b += 32) {
    const int i = b + lane;
    const Tok t = load_tok(scores, modality, c_bits, c_mod, lo, i, whi, nsegs);
    const uint32_t tt = t.seg > 0 ? T[1] : T[0];
    const bool eq = t.seg >= 0 && t.bits == tt;
    const uint32_t em0 = __ballot_sync(0xffffffffu, eq && t.seg == 0);
    const uint32_t em1 = __ballot_sync(0xffffffffu, eq && t.seg == 1);
    bool keep = t.in && (t.seg < 0 || t.bits > tt);
    if (eq) {
      const uint32_t rank = t.seg ? er1 + __popc(em1 & lt_mask) : er0 + __popc(em0 & lt_mask);
      keep = rank < (t.seg ? quota[1] : quota[0]);
    }
    const uint32_t km = __ballot_sync(0xffffffffu, keep);
    const uint32_t p = pos + __popc(km & lt_mask);
    if (t.in) {
      if (keep && p < static_cast<uint32_t>(sq.out_len)) {
        const int o = sq.out_base + static_cast<int>(p);
        keep_idx[o] = i;
        if (modality_out) modality_out[o] = t.mod;
        if (dst_of_src) dst_of_src[i] = o;
      } else if (dst_of_src) {
        dst_of_src[i] = -1;
      }
    }
    pos += __popc(km);
    er0 += __popc(em0);
    er1 += __popc(em1);
  }
}

}  // namespace

template <int CL>
cudaError_t launch_select(const SelectPlan &P, int ns, size_t smem, const float *scores, const uint8_t *modality,
                          int32_t *keep_idx, uint8_t *modality_out, int32_t *dst_of_src, int32_t *new_cu,
                          DeviceError *err, cudaStream_t stream) {
  return launch_pdl(select_kernel<CL>, dim3(CL, ns, 1), dim3(kThreads), smem, stream, P, scores, modality, keep_idx,
                    modality_out, dst_of_src, new_cu, err);
}

// Cluster size per sequence: 8 CTAs, or 16 for sequences longer than kWideFrom tokens where such
// clusters can be resident and every sequence of the launch still gets its own 16 SMs.  Measured
// on GB300 (graph replays, joint top-k): 16 CTAs win from about 30k tokens (26.8 vs 37.2 us at
// 135k), 8 win below (13.3 vs 14.1 us at 16k; 1, 2 or 4 CTAs never win by more than 0.5 us and
// lose up to 11x on long sequences).  0 when the attributes cannot be set.
constexpr int kWideFrom = 24576;

int select_cluster_size(int max_len, int ns) {
  // per device (kernel attributes and residency are properties of the device):
  // 0 = not probed yet, 1 = attributes refused, 2 = 8-CTA clusters, 3 = 16-CTA clusters too
  static std::atomic<int> probed[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  int state = probed[dev].load(std::memory_order_acquire);
  if (state == 0) {
    int ready = 0, large_ok = 0;
    ready = cudaFuncSetAttribute(select_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kCacheBytes)) == cudaSuccess;
    large_ok = ready &&
               cudaFuncSetAttribute(select_kernel<16>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) ==
                   cudaSuccess &&
               cudaFuncSetAttribute(select_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    static_cast<int>(kCacheBytes)) == cudaSuccess;
    if (large_ok) {   // can a 16-CTA cluster of this kernel be resident at all?
      cudaLaunchConfig_t cfg = {};
      cudaLaunchAttribute at[1];
      at[0].id = cudaLaunchAttributeClusterDimension;
      at[0].val.clusterDim.x = 16;
      at[0].val.clusterDim.y = 1;
      at[0].val.clusterDim.z = 1;
      cfg.gridDim = dim3(16, 1, 1);
      cfg.blockDim = dim3(kThreads, 1, 1);
      cfg.dynamicSmemBytes = kCacheBytes;
      cfg.attrs = at;
      cfg.numAttrs = 1;
      int nclusters = 0;
      large_ok = cudaOccupancyMaxActiveClusters(&nclusters, select_kernel<16>, &cfg) == cudaSuccess && nclusters > 0;
    }
    cudaGetLastError();
    state = !ready ? 1 : (large_ok ? 3 : 2);
    probed[dev].store(state, std::memory_order_release);
  }
  if (state == 1) return 0;
  return (max_len > kWideFrom && state == 3 && ns * 16 <= device_sm_count()) ? 16 : 8;
}

apack_status run_select(const apack_seqs *seqs, const float *scores, const int32_t *keep_count_h, int32_t mode,
                        int32_t *keep_idx, uint8_t *modality_out, int32_t *dst_of_src, int32_t *new_cu_seqlens,
                        void *ws, cudaStream_t stream) {
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  if (!keep_count_h || !ws || (mode != APACK_SELECT_PER_MODALITY && mode != APACK_SELECT_JOINT)) return APACK_EINVAL;
  if (T > 0 && (!scores || !keep_idx)) return APACK_EINVAL;
  const int B = seqs->num_seqs;
  const int nsegs = mode == APACK_SELECT_JOINT ? 1 : 2;
  // Host-side plan: counts, output offsets.
  int64_t out_total = 0;
  for (int b = 0; b < B; ++b) {
    const int na = seqs->n_audio_h[b], nv = seqs->n_visual_h[b];
    const int len = seqs->cu_seqlens_h[b + 1] - seqs->cu_seqlens_h[b];
    const int k0 = keep_count_h[2 * b], k1 = keep_count_h[2 * b + 1];
    if (nsegs == 2) {
      if (k0 < 0 || k0 > na || k1 < 0 || k1 > nv) return APACK_EINVAL;
      out_total += len - na - nv + k0 + k1;
    } else {
      if (k0 < 0 || k0 > na + nv) return APACK_EINVAL;
      out_total += len - na - nv + k0;
    }
  }
  (void)out_total;
  const WsLayout L = workspace_layout(seqs);
  DeviceError *err = reinterpret_cast<DeviceError *>(static_cast<uint8_t *>(ws) + L.err_off);
  int32_t out_base = 0;
  for (int s0 = 0; s0 < B; s0 += kSeqsPerLaunch) {
    const int ns = (B - s0 < kSeqsPerLaunch) ? (B - s0) : kSeqsPerLaunch;
    SelectPlan P{};
    P.nseq = ns;
    P.nsegs = nsegs;
    P.write_cu0 = s0 == 0;
    P.seq_base = s0;
    for (int i = 0; i < ns; ++i) {
      const int b = s0 + i;
      SelSeq &q = P.seq[i];
      q.t0 = seqs->cu_seqlens_h[b];
      q.len = seqs->cu_seqlens_h[b + 1] - q.t0;
      const int na = seqs->n_audio_h[b], nv = seqs->n_visual_h[b];
      if (nsegs == 2) {
        q.n_seg[0] = na; q.n_seg[1] = nv;
        q.k[0] = keep_count_h[2 * b]; q.k[1] = keep_count_h[2 * b + 1];
      } else {
        q.n_seg[0] = na + nv; q.n_seg[1] = 0;
        q.k[0] = keep_count_h[2 * b]; q.k[1] = 0;
      }
      q.out_len = q.len - na - nv + q.k[0] + q.k[1];
      q.out_base = out_base;
      out_base += q.out_len;
    }
    int max_len = 0;
    for (int i = 0; i < ns; ++i) max_len = P.seq[i].len > max_len ? P.seq[i].len : max_len;
    const int CL = select_cluster_size(max_len, ns);
    if (CL == 0) return APACK_ECUDA;
    // cache each CTA's slice in shared memory when the longest slice of the launch fits
    const int slice = (max_len + CL - 1) / CL;
    size_t smem = 0;
    if (slice <= kMaxCached) {
      P.cache_tokens = slice;
      smem = static_cast<size_t>(slice) * 5;
    }
    cudaError_t e = cudaSuccess;
    if (CL == 16)
      e = launch_select<16>(P, ns, smem, scores, seqs->modality, keep_idx, modality_out, dst_of_src, new_cu_seqlens,
                            err, stream);
    else
      e = launch_select<8>(P, ns, smem, scores, seqs->modality, keep_idx, modality_out, dst_of_src, new_cu_seqlens,
                           err, stream);
    if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  return APACK_OK;
}

}  // namespace apack
