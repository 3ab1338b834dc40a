// select.cu -- per-(sequence, modality) top-k of Eq. inner (Sec. 3.2) and the stable keep map.
//
// One thread-block cluster of kCluster CTAs per sequence; CTA c owns a
// contiguous slice of the sequence's tokens.
//
//  1. Radix select (4 passes of 8 bits, most significant first) of the k-th
//     largest score of every segment.  Scores are >= 0, so the order of their
//     IEEE bit patterns as unsigned integers is their numeric order.  Each CTA
//     builds a shared-memory histogram of its slice; the cluster merges them
//     through distributed shared memory and every CTA derives the same digit.
//     The result per segment is a threshold bit pattern T and a quota q: keep
//     every score > T and the first q scores == T in token order (ties go to
//     the lower index).
//  2. Counts per CTA (other tokens, > T, == T) are exchanged through DSMEM so
//     that each CTA knows its output offset and how many ties precede it.
//  3. Each CTA walks its slice in token order with block-wide scans and writes
//     keep_idx (ascending), the compacted modality and dst_of_src.
#include <cstdio>

#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kCluster = 8;
constexpr int kThreads = 512;
constexpr int kWarps = kThreads / 32;
constexpr int kItems = 8;                       // contiguous tokens per thread per tile
constexpr int kTile = kThreads * kItems;

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
  SelSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int seg_of(uint8_t m, int nsegs) {
  if (m == APACK_MOD_AUDIO) return 0;
  if (m == APACK_MOD_VISUAL) return nsegs == 1 ? 0 : 1;
  return -1;
}

// Exclusive block scan of one uint32 per thread; returns the exclusive prefix
// and writes the block total to *total.  Uses `scratch` [kWarps + 1].
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t *scratch, uint32_t *total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t incl = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t n = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += n;
  }
  if (lane == 31) scratch[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    uint32_t w = lane < kWarps ? scratch[lane] : 0u;
    uint32_t wi = w;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const uint32_t n = __shfl_up_sync(0xffffffffu, wi, off);
      if (lane >= off) wi += n;
    }
    if (lane < kWarps) scratch[lane] = wi - w;       // exclusive warp offsets
    if (lane == kWarps - 1) scratch[kWarps] = wi;    // block total
  }
  __syncthreads();
  const uint32_t res = scratch[warp] + incl - v;
  *total = scratch[kWarps];
  __syncthreads();
  return res;
}

// Loads the kItems contiguous tokens of this thread in the tile at `base`
// (segment -1 and bits 0 past `hi` or outside S).  All loads are issued
// before any is used.
__device__ __forceinline__ void load_items(const float *__restrict__ scores, const uint8_t *__restrict__ modality,
                                           int base, int hi, int nsegs, int (&seg)[kItems],
                                           uint32_t (&bits)[kItems], uint8_t (&mod)[kItems]) {
  const int i0 = base + threadIdx.x * kItems;
#pragma unroll
  for (int j = 0; j < kItems; ++j) {
    const bool in = i0 + j < hi;
    mod[j] = in ? modality[i0 + j] : static_cast<uint8_t>(0xFF);
    bits[j] = in ? __float_as_uint(scores[i0 + j]) : 0u;
  }
#pragma unroll
  for (int j = 0; j < kItems; ++j) seg[j] = seg_of(mod[j], nsegs);
}

__global__ void __cluster_dims__(kCluster, 1, 1) __launch_bounds__(kThreads)
    select_kernel(const __grid_constant__ SelectPlan plan, const float *__restrict__ scores,
                  const uint8_t *__restrict__ modality, int32_t *__restrict__ keep_idx,
                  uint8_t *__restrict__ modality_out, int32_t *__restrict__ dst_of_src,
                  int32_t *__restrict__ new_cu, DeviceError *err) {
  __shared__ uint32_t hist[2][2][256];
  __shared__ uint32_t st_prefix[2], st_mask[2], st_krem[2], st_total[2];
  __shared__ uint32_t cnt[5];                 // other, gt0, gt1, eq0, eq1 (read by the cluster)
  __shared__ uint32_t scratch[kWarps + 1];
  __shared__ int32_t info[6];                 // kept_before, eq_before0, eq_before1, eq_mode0, eq_mode1

  const SelSeq &sq = plan.seq[blockIdx.y];
  const uint32_t crank = cluster_ctarank();
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int nsegs = plan.nsegs;
  const int chunk = (sq.len + kCluster - 1) / kCluster;
  const int lo = sq.t0 + min(sq.len, static_cast<int>(crank) * chunk);
  const int hi = sq.t0 + min(sq.len, static_cast<int>(crank + 1) * chunk);

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
    for (int base = lo; base < hi; base += kTile) {
      int sg[kItems];
      uint32_t bt[kItems];
      uint8_t md[kItems];
      load_items(scores, modality, base, hi, nsegs, sg, bt, md);
#pragma unroll
      for (int j = 0; j < kItems; ++j) {
        if (sg[j] < 0) continue;
        const uint32_t pm = sg[j] ? p1 : p0, mm = sg[j] ? m1 : m0;
        if ((bt[j] & mm) == pm) atomicAdd(&hist[hb][sg[j]][(bt[j] >> shift) & 255u], 1u);
      }
    }
    __syncthreads();
    cluster_sync();
    for (int j = tid; j < 2 * 256; j += kThreads) (&hist[hb ^ 1][0][0])[j] = 0u;
    if (warp < nsegs) {
      const int seg = warp;
      uint32_t c[8];
      uint32_t lsum = 0;
#pragma unroll
      for (int b = 0; b < 8; ++b) {
        uint32_t v = 0;
        for (int r = 0; r < kCluster; ++r)
          v += ld_shared_cluster_u32(map_shared_rank(&hist[hb][seg][lane * 8 + b], r));
        c[b] = v;
        lsum += v;
      }
      // inclusive suffix sum over lanes (higher lanes hold higher digits)
      uint32_t suf = lsum;
#pragma unroll
      for (int off = 1; off < 32; off <<= 1) {
        const uint32_t n = __shfl_down_sync(0xffffffffu, suf, off);
        if (lane + off < 32) suf += n;
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

  // ---- 2. per-CTA counts, exchanged through the cluster
  {
    uint32_t other = 0, gt0 = 0, gt1 = 0, eq0 = 0, eq1 = 0;
    for (int base = lo; base < hi; base += kTile) {
      int sg[kItems];
      uint32_t bt[kItems];
      uint8_t md[kItems];
      load_items(scores, modality, base, hi, nsegs, sg, bt, md);
#pragma unroll
      for (int j = 0; j < kItems; ++j) {
        if (base + tid * kItems + j >= hi) break;
        if (sg[j] < 0) { ++other; continue; }
        const uint32_t t = sg[j] ? T[1] : T[0];
        if (bt[j] > t) { if (sg[j]) ++gt1; else ++gt0; }
        else if (bt[j] == t) { if (sg[j]) ++eq1; else ++eq0; }
      }
    }
    uint32_t tot;
    // five reductions through the scan helper (exclusive value unused)
    block_exclusive_scan(other, scratch, &tot); if (tid == 0) cnt[0] = tot;
    block_exclusive_scan(gt0, scratch, &tot);   if (tid == 0) cnt[1] = tot;
    block_exclusive_scan(gt1, scratch, &tot);   if (tid == 0) cnt[2] = tot;
    block_exclusive_scan(eq0, scratch, &tot);   if (tid == 0) cnt[3] = tot;
    block_exclusive_scan(eq1, scratch, &tot);   if (tid == 0) cnt[4] = tot;
  }
  __syncthreads();
  cluster_sync();
  if (tid == 0) {
    uint32_t kept_before = 0, eqb[2] = {0, 0}, kept_all = 0, seg_dev[2] = {0, 0};
    // Walk the CTAs in order: ties are granted to CTAs until the quota runs out.
    uint32_t eq_prefix[2] = {0, 0};
    for (int r = 0; r < kCluster; ++r) {
      uint32_t c[5];
      for (int j = 0; j < 5; ++j) c[j] = ld_shared_cluster_u32(map_shared_rank(&cnt[j], r));
      uint32_t kept = c[0] + c[1] + c[2];
      for (int s = 0; s < 2; ++s) {
        const uint32_t ties = c[3 + s];
        const uint32_t avail = quota[s] > eq_prefix[s] ? quota[s] - eq_prefix[s] : 0u;
        kept += ties < avail ? ties : avail;
        seg_dev[s] += c[1 + s] + ties;
        if (r == static_cast<int>(crank)) eqb[s] = eq_prefix[s];
        eq_prefix[s] += ties;
      }
      if (r < static_cast<int>(crank)) kept_before += kept;
      kept_all += kept;
    }
    info[0] = static_cast<int32_t>(kept_before);
    for (int s = 0; s < 2; ++s) {
      info[1 + s] = static_cast<int32_t>(eqb[s]);
      // tie mode of this CTA: 0 = drop all its ties, 1 = keep all, 2 = rank them
      const uint32_t my_ties = cnt[3 + s];
      int mode;
      if (eqb[s] >= quota[s]) mode = 0;
      else if (eqb[s] + my_ties <= quota[s]) mode = 1;
      else mode = 2;
      info[3 + s] = mode;
    }
    if (crank == 0) {
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

  // ---- 3. ordered write of the kept tokens of this slice
  uint32_t run_keep = static_cast<uint32_t>(info[0]);
  uint32_t run_eq[2] = {static_cast<uint32_t>(info[1]), static_cast<uint32_t>(info[2])};
  const int mode0 = info[3], mode1 = info[4];
  const bool need_rank = (mode0 == 2) || (mode1 == 2);
  for (int base = lo; base < hi; base += kTile) {
    int sg[kItems];
    uint32_t bt[kItems];
    uint8_t md[kItems];
    load_items(scores, modality, base, hi, nsegs, sg, bt, md);
    const int i0 = base + tid * kItems;
    bool keep[kItems], eq[kItems];
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      const bool valid = i0 + j < hi;
      const uint32_t t = sg[j] > 0 ? T[1] : T[0];
      eq[j] = valid && sg[j] >= 0 && bt[j] == t;
      keep[j] = valid && (sg[j] < 0 || bt[j] > t || (eq[j] && (sg[j] ? mode1 : mode0) == 1));
    }
    if (need_rank) {
      // ties ranked in token order: per-thread counts (packed: low 16 bits
      // segment 0, high 16 bits segment 1), then a block scan
      uint32_t e = 0;
#pragma unroll
      for (int j = 0; j < kItems; ++j)
        if (eq[j]) e += sg[j] ? (1u << 16) : 1u;
      uint32_t etot;
      uint32_t ex = block_exclusive_scan(e, scratch, &etot);
      uint32_t r0 = run_eq[0] + (ex & 0xFFFFu), r1 = run_eq[1] + (ex >> 16);
#pragma unroll
      for (int j = 0; j < kItems; ++j) {
        if (!eq[j]) continue;
        const int md2 = sg[j] ? mode1 : mode0;
        uint32_t &r = sg[j] ? r1 : r0;
        if (md2 == 2) keep[j] = r < (sg[j] ? quota[1] : quota[0]);
        ++r;
      }
      run_eq[0] += etot & 0xFFFFu;
      run_eq[1] += etot >> 16;
    }
    uint32_t nk = 0;
#pragma unroll
    for (int j = 0; j < kItems; ++j) nk += keep[j] ? 1u : 0u;
    uint32_t ktot;
    uint32_t pos = run_keep + block_exclusive_scan(nk, scratch, &ktot);
#pragma unroll
    for (int j = 0; j < kItems; ++j) {
      if (i0 + j >= hi) break;
      if (keep[j] && pos < static_cast<uint32_t>(sq.out_len)) {
        const int o = sq.out_base + static_cast<int>(pos);
        keep_idx[o] = i0 + j;
        if (modality_out) modality_out[o] = md[j];
        if (dst_of_src) dst_of_src[i0 + j] = o;
      } else if (dst_of_src) {
        dst_of_src[i0 + j] = -1;
      }
      if (keep[j]) ++pos;
    }
    run_keep += ktot;
  }
}

}  // namespace

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
    dim3 grid(kCluster, ns, 1);
    select_kernel<<<grid, kThreads, 0, stream>>>(P, scores, seqs->modality, keep_idx, modality_out, dst_of_src,
                                                 new_cu_seqlens, err);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  return APACK_OK;
}

}  // namespace apack
