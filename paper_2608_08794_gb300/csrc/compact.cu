// compact.cu -- KV-cache and hidden-state slicing of Sec. 3.2 (Algorithm 1, "slice their
// KV-cache entries"): dst row j = src row keep_idx[j] for every plane.
//
// HBM-bound: every byte is read once and written once.
//  - TMA kernel (rows of 16-byte multiples up to 32 KB, 16-byte aligned): one
//    warp per CTA streams kept rows into a ring of 32 KB shared-memory slots
//    with cp.async.bulk (one row per lane, completion on the slot's mbarrier)
//    and writes each slot back with a single bulk store when the output rows
//    are contiguous (one per row otherwise).  Several slots stay in flight per
//    CTA, so a handful of threads keep the whole HBM pipe busy.
//  - Rows that are not 16-byte multiples (or misaligned) take the narrow
//    kernel, one thread per row.
//  - In place (src == dst): output row j reads row keep_idx[j] >= j, so the
//    store of output rows [r0, r0 + n) of a plane may only start once every
//    load of that plane that reads a row in [r0, r0 + n) is done.  Those loads
//    belong to output rows below r0 + n: earlier items of the same plane.
//    The in-place kernel runs two CTAs per SM (cooperative launch, so
//    all are resident), items round-robin as in the out-of-place kernel; each
//    CTA publishes how many of its items' loads are complete, and waits
//    (bounded) for the owners of those earlier items before each store.
//    Loads never wait on stores of later items, so the waits always end.
#include "internal.cuh"
#include "ptx.cuh"

namespace apack {

namespace {

constexpr int kMaxGroups = 16;
constexpr int kSlots = 3;                       // slots per CTA (two CTAs per SM)
constexpr uint32_t kSlotBytes = 32768;
constexpr uint32_t kTmaSmem = kSlots * kSlotBytes;

struct TmaGroup {
  const uint8_t *src;
  uint8_t *dst;
  int64_t sps, dps, srs, drs;   // plane and row strides in bytes
  uint32_t row_bytes;
  uint32_t rows_per_slot;
  uint32_t chunks_per_plane;    // ceil(n_out / rows_per_slot)
  uint32_t item_begin;          // first slot-sized item of this group
  uint32_t contiguous;          // output rows are back to back (one bulk store per slot)
  uint32_t chunk_major;         // items ordered (chunk, plane) instead of (plane, chunk): in place
  uint32_t num_planes;
  uint32_t pad;
};

struct TmaPlan {
  int32_t ngroups;
  uint32_t total_items;
  uint32_t n_out;
  uint32_t dep_period;          // in place: owners of a plane's items repeat after this many chunks
  TmaGroup g[kMaxGroups];
};

struct Item {
  const TmaGroup *grp;
  uint32_t plane, r0, nrows;
};

__device__ __forceinline__ Item decode_item(const TmaPlan &p, uint32_t item) {
  int gi = 0;
  while (gi + 1 < p.ngroups && p.g[gi + 1].item_begin <= item) ++gi;
  const TmaGroup &G = p.g[gi];
  const uint32_t local = item - G.item_begin;
  Item it;
  it.grp = &G;
  uint32_t chunk;
  if (G.chunk_major) {
    chunk = local / G.num_planes;
    it.plane = local - chunk * G.num_planes;
  } else {
    it.plane = local / G.chunks_per_plane;
    chunk = local - it.plane * G.chunks_per_plane;
  }
  it.r0 = chunk * G.rows_per_slot;
  it.nrows = min(G.rows_per_slot, p.n_out - it.r0);
  return it;
}

// Loads the kept rows of one item into a slot (all lanes take part).
__device__ __forceinline__ void load_item(const Item &it, uint8_t *slot, uint64_t *bar,
                                          const int32_t *__restrict__ keep_idx, int lane) {
  const TmaGroup &G = *it.grp;
  if (lane == 0) mbar_arrive_expect_tx(bar, it.nrows * G.row_bytes);
  __syncwarp();
  const uint8_t *src = G.src + static_cast<int64_t>(it.plane) * G.sps;
  for (uint32_t r = lane; r < it.nrows; r += 32) {
    const int64_t srow = keep_idx[it.r0 + r];
    bulk_load(slot + r * G.row_bytes, src + srow * G.srs, G.row_bytes, bar);
  }
}

// Stores a full slot to the output rows of its item; every lane commits its group.
__device__ __forceinline__ void store_item(const Item &it, const uint8_t *slot, int lane) {
  const TmaGroup &G = *it.grp;
  uint8_t *dst = G.dst + static_cast<int64_t>(it.plane) * G.dps + static_cast<int64_t>(it.r0) * G.drs;
  if (G.contiguous) {
    if (lane == 0) bulk_store(dst, slot, it.nrows * G.row_bytes);
  } else {
    for (uint32_t r = lane; r < it.nrows; r += 32) bulk_store(dst + r * G.drs, slot + r * G.row_bytes, G.row_bytes);
  }
  bulk_commit();
}

__global__ void __launch_bounds__(32) gather_tma_kernel(const __grid_constant__ TmaPlan plan,
                                                        const int32_t *__restrict__ keep_idx, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t slots[];
  __shared__ __align__(8) uint64_t full[kSlots];
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int i = 0; i < kSlots; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  __syncwarp();
  // this CTA's items: blockIdx.x, blockIdx.x + gridDim.x, ...
  const uint32_t first = blockIdx.x, stride = gridDim.x;
  const uint32_t n_mine = first < plan.total_items ? (plan.total_items - first + stride - 1) / stride : 0;
  uint32_t issued = n_mine < kSlots ? n_mine : kSlots;   // positions whose loads were issued
  for (uint32_t j = 0; j < issued; ++j)
    load_item(decode_item(plan, first + j * stride), slots + j * kSlotBytes, &full[j], keep_idx, lane);
  bool ok = true;
  uint32_t j = 0;
  for (; j < n_mine; ++j) {
    const int slot = j % kSlots;
    const Item it = decode_item(plan, first + j * stride);
    if (!mbar_wait(&full[slot], (j / kSlots) & 1u, kWaitLimitNs)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 41);
      ok = false;
      break;
    }
    fence_proxy_async_smem();
    store_item(it, slots + slot * kSlotBytes, lane);
    // refill the slot whose store was issued one item ago, once that store has read it
    if (j >= 1 && j - 1 + kSlots < n_mine) {
      bulk_wait_read<1>();
      const uint32_t k = j - 1 + kSlots;
      const int ks = k % kSlots;
      load_item(decode_item(plan, first + k * stride), slots + ks * kSlotBytes, &full[ks], keep_idx, lane);
      issued = k + 1;
    }
  }
  if (!ok) {
    // loads of items j .. issued - 1 may still be in flight: wait for them (bounded)
    for (uint32_t k = j; k < issued; ++k) mbar_wait(&full[k % kSlots], (k / kSlots) & 1u, kWaitLimitNs / 4);
  }
  bulk_wait_all();
}

// ------------------------------------------------------------------ in place
constexpr int kInSlots = 3;                      // two CTAs per SM, 3 slots of 32 KB each
constexpr uint32_t kInSmem = kInSlots * kSlotBytes;
constexpr int kMaxInCtas = 384;                  // 16-bit progress words at ws + 256 .. ws + 1024
constexpr int kInChecks = 384;                   // progress words one dependency check may read
constexpr size_t kProgressOff = 256;

// Progress words.  A word is written after the CTA has observed its loads complete (the rows are
// already in shared memory, so no later write can change what they read), and a reader only
// issues its store after the loop that reads the word has seen the value it needs: relaxed
// gpu-scope accesses carry all the ordering the stores need.
__device__ __forceinline__ uint32_t ld_progress(const uint16_t *p) {
  uint16_t v;
  asm volatile("ld.relaxed.gpu.global.u16 %0, [%1];" : "=h"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void st_progress(uint16_t *p, uint32_t v) {
  asm volatile("st.relaxed.gpu.global.u16 [%0], %1;" ::"l"(p), "h"(static_cast<uint16_t>(v)) : "memory");
}

// #{ r < n : a[r] < x } for a strictly increasing, given a bracket [lo, hi] that holds it
// (a[lo - 1] < x or lo == 0; hi == n or a[hi] >= x).  Rounds of 32 evenly spaced probes narrow
// wide brackets; a bracket of at most 256 rows is then counted in one round, 8 rows per lane
// (independent loads of a few adjacent cache lines).
constexpr uint32_t kCountRows = 8;

__device__ __forceinline__ uint32_t warp_count_below(const int32_t *__restrict__ a, uint32_t lo, uint32_t hi,
                                                     int64_t x, int lane) {
  while (hi - lo > 32 * kCountRows) {
    const uint32_t span = hi - lo;
    const uint32_t step = (span + 31) / 32;
    const uint32_t p = lo + lane * step;
    const uint32_t b = __ballot_sync(0xffffffffu, p < hi && a[p] >= x);
    if (b) {
      const int f = __ffs(b) - 1;
      hi = lo + f * step;
      if (f > 0) lo += (f - 1) * step + 1;
    } else {
      lo += ((span - 1) / step) * step + 1;                 // past the last probe inside [lo, hi)
    }
  }
  uint32_t cnt = 0;
  const uint32_t p0 = lo + lane * kCountRows;
#pragma unroll
  for (uint32_t i = 0; i < kCountRows; ++i) cnt += (p0 + i < hi && a[p0 + i] < x) ? 1u : 0u;
  return lo + __reduce_add_sync(0xffffffffu, cnt);
}

__global__ void __launch_bounds__(32) gather_inplace_kernel(const __grid_constant__ TmaPlan plan,
                                                            const int32_t *__restrict__ keep_idx,
                                                            uint16_t *progress, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t slots[];
  __shared__ __align__(8) uint64_t full[kInSlots];
  __shared__ uint16_t seen[kMaxInCtas];          // last progress read of every CTA
  const int lane = threadIdx.x;
  if (lane == 0) {
    for (int i = 0; i < kInSlots; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  for (int i = lane; i < kMaxInCtas; i += 32) seen[i] = 0;
  __syncwarp();
  const uint32_t me = blockIdx.x, P = gridDim.x;
  const uint32_t n_mine = me < plan.total_items ? (plan.total_items - me + P - 1) / P : 0;
  uint32_t issued = n_mine < kInSlots ? n_mine : kInSlots;   // positions whose loads were issued
  for (uint32_t j = 0; j < issued; ++j)
    load_item(decode_item(plan, me + j * P), slots + j * kSlotBytes, &full[j], keep_idx, lane);
  bool ok = true;
  uint32_t waited = 0;                                        // positions whose loads were observed
  uint32_t hint_row = 0;                                      // #{ keep_idx < hint_limit }, previous item
  int64_t hint_limit = 0;
  const TmaGroup *hint_grp = nullptr;
  for (uint32_t j = 0; ok && j < n_mine; ++j) {
    const int slot = j % kInSlots;
    const uint32_t item = me + j * P;
    const Item it = decode_item(plan, item);
    if (j >= waited && !mbar_wait(&full[slot], (j / kInSlots) & 1u, kWaitLimitNs)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 42);
      ok = false;
      break;
    }
    // publish as far as the loads are complete: this item, and the next ones already landed
    if (j >= waited) {
      uint32_t w = j + 1;
      if (lane == 0) {
        while (w < issued && mbar_try_wait(&full[w % kInSlots], (w / kInSlots) & 1u)) ++w;
        st_progress(progress + me, w);
      }
      waited = __shfl_sync(0xffffffffu, w, 0);              // the same count in every lane
    }
    // items of this plane whose loads read rows [r0, r0 + n) hold the output rows whose source is
    // below r0 + n: chunks <= c_hi, the chunk of the last such row (far behind c once rows are
    // dropped, so these waits are mostly met already).  Those are items item - k * num_planes,
    // k >= c - c_hi; their owners repeat with period P / gcd(num_planes, P) in k and an owner's
    // progress is monotonic, so the first period covers them all (at most kInChecks words).
    const TmaGroup &G = *it.grp;
    const uint32_t c = it.r0 / G.rows_per_slot;
    const int64_t limit = static_cast<int64_t>(it.r0) + it.nrows;
    {
      // keep_idx holds distinct integers, so the count below limit grows by at most limit -
      // hint_limit from the previous item of the group, and never exceeds limit
      const int64_t n = plan.n_out;
      const bool same = &G == hint_grp;
      const uint32_t lo = same ? hint_row : 0;
      const uint32_t hi = static_cast<uint32_t>(same ? min(n, static_cast<int64_t>(hint_row) + (limit - hint_limit))
                                                     : min(n, limit));
      hint_row = warp_count_below(keep_idx, lo, hi, limit, lane);
      hint_limit = limit;
      hint_grp = &G;
    }
    uint32_t kmin = 1, kmax = 0;                          // no dependency unless some row reads below limit
    if (hint_row > 0) {
      const uint32_t c_hi = (hint_row - 1) / G.rows_per_slot;
      kmin = c > c_hi ? c - c_hi : 1;
      kmax = min(c, kmin + plan.dep_period - 1);
    }
    uint32_t owner[kInChecks / 32], need[kInChecks / 32];
    {
      // item - k * num_planes for k = kmin + lane + 32 u: one division, then steps of 32 planes
      const uint32_t d = 32u * G.num_planes, dq = d / P, dr = d - dq * P;
      const uint32_t other0 = item - (kmin + lane) * G.num_planes;   // only used while k <= kmax
      uint32_t o = other0 % P, q = other0 / P;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) {
        const uint32_t k = kmin + lane + 32 * u;
        owner[u] = me;                                    // no check: my own items are waited in order
        need[u] = 0;
        if (k <= kmax) {
          owner[u] = o;
          need[u] = q + 1;
        }
        // the next u: other - d
        const bool borrow = o < dr;
        o = borrow ? o + P - dr : o - dr;
        q = q - dq - (borrow ? 1u : 0u);
      }
    }
    // each lane owns distinct owners (k differ by less than the period), so the cache needs no sync.
    // When any cached word is too old, every owner of the check is read again in the same round:
    // the words read are far ahead of what later items need, so the cache then lasts until the
    // needs have grown past them (a few rounds per launch instead of one per stale owner).
    bool mine_ok = true;
    uint64_t t0 = 0;                                      // the clock is read once a round has failed
    for (;;) {
      bool stale = false;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) stale |= owner[u] != me && seen[owner[u]] < need[u];
      if (!__any_sync(0xffffffffu, stale)) break;
      bool all = true;
#pragma unroll
      for (int u = 0; u < kInChecks / 32; ++u) {
        if (owner[u] != me) {
          const uint32_t v = ld_progress(progress + owner[u]);
          seen[owner[u]] = v;
          all &= v >= need[u];
        }
      }
      if (__all_sync(0xffffffffu, all)) break;
      if (t0 == 0) t0 = globaltimer_ns();
      if (__any_sync(0xffffffffu, globaltimer_ns() - t0 > kWaitLimitNs)) {   // the warp gives up together
        mine_ok = false;
        break;
      }
    }
    if (!__all_sync(0xffffffffu, mine_ok)) {
      if (lane == 0 && err) raise_device_error(err, APACK_ETIMEOUT, 43);
      ok = false;
      break;
    }
    asm volatile("fence.proxy.async.global;" ::: "memory");   // the observed loads before the bulk store
    fence_proxy_async_smem();
    store_item(it, slots + slot * kSlotBytes, lane);
    if (j >= 1 && j - 1 + kInSlots < n_mine) {
      bulk_wait_read<1>();
      const uint32_t k = j - 1 + kInSlots;
      const int ks = k % kInSlots;
      load_item(decode_item(plan, me + k * P), slots + ks * kSlotBytes, &full[ks], keep_idx, lane);
      issued = k + 1;
    }
  }
  if (!ok) {
    // loads issued but not observed may still be in flight: wait for them (bounded)
    for (uint32_t k = waited; k < issued; ++k) mbar_wait(&full[k % kInSlots], (k / kInSlots) & 1u, kWaitLimitNs / 4);
  }
  bulk_wait_all();
}

// ------------------------------------------------------------------ host source
// Source rows in pinned host memory (zero copy): only the kept rows cross the host link.
// Consecutive threads take consecutive 16-byte pieces of a row (coalesced link reads); each
// thread issues U loads before its U stores so that enough reads are in flight.
constexpr int kHostUnroll = 4;

__global__ void __launch_bounds__(256) gather_host_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst,
                                                          int64_t sps, int64_t dps, int64_t srs, int64_t drs,
                                                          int64_t row_bytes, int64_t n_planes, int64_t n_out,
                                                          const int32_t *__restrict__ keep_idx) {
  const int64_t vec_per_row = row_bytes / 16;
  const int64_t total = n_planes * n_out * vec_per_row;
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t base = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; base < total;
       base += stride * kHostUnroll) {
    uint4 v[kHostUnroll];
#pragma unroll
    for (int u = 0; u < kHostUnroll; ++u) {
      const int64_t e = base + u * stride;
      if (e < total) {
        const int64_t row = e / vec_per_row, c = e - row * vec_per_row;
        const int64_t plane = row / n_out, j = row - plane * n_out;
        v[u] = *reinterpret_cast<const uint4 *>(src + plane * sps + static_cast<int64_t>(keep_idx[j]) * srs + c * 16);
      }
    }
#pragma unroll
    for (int u = 0; u < kHostUnroll; ++u) {
      const int64_t e = base + u * stride;
      if (e < total) {
        const int64_t row = e / vec_per_row, c = e - row * vec_per_row;
        const int64_t plane = row / n_out, j = row - plane * n_out;
        *reinterpret_cast<uint4 *>(dst + plane * dps + j * drs + c * 16) = v[u];
      }
    }
  }
}

// Device address of a pinned host buffer, or nullptr when src is not host memory.
const void *host_source(const void *src) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, src) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return at.type == cudaMemoryTypeHost ? at.devicePointer : nullptr;
}

// One thread per (plane, row); copies with the widest access the row allows.
__global__ void gather_narrow_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst, int64_t sps,
                                     int64_t dps, int64_t srs, int64_t drs, int64_t row_bytes, int unit,
                                     int64_t n_planes, int64_t n_out, const int32_t *__restrict__ keep_idx) {
  const int64_t t = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  if (t >= n_planes * n_out) return;
  const int64_t plane = t / n_out, row = t - plane * n_out;
  const uint8_t *s = src + plane * sps + static_cast<int64_t>(keep_idx[row]) * srs;
  uint8_t *d = dst + plane * dps + row * drs;
  switch (unit) {
    case 16:
      for (int64_t b = 0; b < row_bytes; b += 16)
        *reinterpret_cast<uint4 *>(d + b) = *reinterpret_cast<const uint4 *>(s + b);
      break;
    case 8:
      for (int64_t b = 0; b < row_bytes; b += 8)
        *reinterpret_cast<uint2 *>(d + b) = *reinterpret_cast<const uint2 *>(s + b);
      break;
    case 4:
      for (int64_t b = 0; b < row_bytes; b += 4)
        *reinterpret_cast<uint32_t *>(d + b) = *reinterpret_cast<const uint32_t *>(s + b);
      break;
    case 2:
      for (int64_t b = 0; b < row_bytes; b += 2)
        *reinterpret_cast<uint16_t *>(d + b) = *reinterpret_cast<const uint16_t *>(s + b);
      break;
    default:
      for (int64_t b = 0; b < row_bytes; ++b) d[b] = s[b];
  }
}

int widest_unit(const apack_plane &p) {
  const uint64_t bits = reinterpret_cast<uintptr_t>(p.src) | reinterpret_cast<uintptr_t>(p.dst) |
                        static_cast<uint64_t>(p.src_plane_stride) | static_cast<uint64_t>(p.dst_plane_stride) |
                        static_cast<uint64_t>(p.src_row_stride) | static_cast<uint64_t>(p.dst_row_stride) |
                        static_cast<uint64_t>(p.row_bytes);
  for (int u = 16; u > 1; u >>= 1)
    if ((bits & static_cast<uint64_t>(u - 1)) == 0) return u;
  return 1;
}

bool ranges_overlap(const apack_plane &p, int64_t n_rows_src, int64_t n_out) {
  const uint8_t *s0 = static_cast<const uint8_t *>(p.src);
  const uint8_t *d0 = static_cast<const uint8_t *>(p.dst);
  const int64_t s_span = (p.num_planes - 1) * p.src_plane_stride + (n_rows_src - 1) * p.src_row_stride + p.row_bytes;
  const int64_t d_span = (p.num_planes - 1) * p.dst_plane_stride + (n_out - 1) * p.dst_row_stride + p.row_bytes;
  return s0 < d0 + d_span && d0 < s0 + s_span;
}

}  // namespace

apack_status run_compact(const int32_t *keep_idx, int64_t n_out, const apack_plane *planes, int32_t num_groups,
                         DeviceError *err, cudaStream_t stream) {
  if (n_out < 0 || num_groups < 0 || (num_groups > 0 && !planes)) return APACK_EINVAL;
  if (n_out == 0 || num_groups == 0) return APACK_OK;
  if (!keep_idx || n_out > INT32_MAX) return APACK_EINVAL;
  // validate and plan every group before anything touches the device
  TmaPlan tp{}, ip{};           // out-of-place groups, in-place groups
  tp.n_out = ip.n_out = static_cast<uint32_t>(n_out);
  uint64_t items = 0, in_items = 0;
  int narrow[kMaxGroups * 4];
  int n_narrow = 0;
  apack_plane host_groups[kMaxGroups * 4];
  int n_host = 0;
  for (int i = 0; i < num_groups; ++i) {
    const apack_plane &p = planes[i];
    if (p.num_planes < 0 || p.row_bytes < 0) return APACK_EINVAL;
    if (p.num_planes == 0 || p.row_bytes == 0) continue;
    if (!p.src || !p.dst || p.src_row_stride < p.row_bytes || p.dst_row_stride < p.row_bytes ||
        p.src_plane_stride < 0 || p.dst_plane_stride < 0)
      return APACK_EINVAL;
    const bool tma_rows = widest_unit(p) == 16 && p.row_bytes <= static_cast<int64_t>(kSlotBytes);
    if (const void *hs = host_source(p.src)) {
      // pinned host source: zero-copy gather (destination in device memory, never in place)
      if (p.src == p.dst || host_source(p.dst)) return APACK_EINVAL;
      if (n_host == kMaxGroups * 4) return APACK_EINVAL;
      host_groups[n_host] = p;
      host_groups[n_host].src = hs;
      ++n_host;
      continue;
    }
    if (p.src == p.dst) {
      // in place: same layout on both sides, vector rows, and the progress words of the workspace
      if (p.src_plane_stride != p.dst_plane_stride || p.src_row_stride != p.dst_row_stride) return APACK_EINVAL;
      if (!tma_rows) return APACK_EUNSUPPORTED;
      if (!err) return APACK_EINVAL;
    } else if (ranges_overlap(p, n_out, n_out)) {
      return APACK_EINVAL;
    }
    if (tma_rows) {
      TmaPlan &pl = p.src == p.dst ? ip : tp;
      uint64_t &cnt = p.src == p.dst ? in_items : items;
      if (pl.ngroups == kMaxGroups) return APACK_EINVAL;
      TmaGroup &g = pl.g[pl.ngroups++];
      g.src = static_cast<const uint8_t *>(p.src);
      g.dst = static_cast<uint8_t *>(p.dst);
      g.sps = p.src_plane_stride;
      g.dps = p.dst_plane_stride;
      g.srs = p.src_row_stride;
      g.drs = p.dst_row_stride;
      g.row_bytes = static_cast<uint32_t>(p.row_bytes);
      g.rows_per_slot = kSlotBytes / g.row_bytes;
      g.chunks_per_plane = static_cast<uint32_t>((n_out + g.rows_per_slot - 1) / g.rows_per_slot);
      g.item_begin = static_cast<uint32_t>(cnt);
      g.contiguous = p.dst_row_stride == p.row_bytes;
      g.chunk_major = p.src == p.dst;
      g.num_planes = static_cast<uint32_t>(p.num_planes);
      cnt += static_cast<uint64_t>(g.chunks_per_plane) * p.num_planes;
      if (cnt > 0x7FFFFFFFull) return APACK_EINVAL;
    } else {
      if (n_narrow == kMaxGroups * 4) return APACK_EINVAL;
      narrow[n_narrow++] = i;
    }
  }
  for (int k = 0; k < n_host; ++k) {
    const apack_plane &p = host_groups[k];
    if (widest_unit(p) == 16) {
      const int64_t n = static_cast<int64_t>(p.num_planes) * n_out * (p.row_bytes / 16);
      int64_t blocks = (n + 256 * kHostUnroll - 1) / (256 * kHostUnroll);
      const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
      if (blocks > cap) blocks = cap;
      gather_host_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
          static_cast<const uint8_t *>(p.src), static_cast<uint8_t *>(p.dst), p.src_plane_stride, p.dst_plane_stride,
          p.src_row_stride, p.dst_row_stride, p.row_bytes, p.num_planes, n_out, keep_idx);
    } else {
      const int64_t n = static_cast<int64_t>(p.num_planes) * n_out;
      gather_narrow_kernel<<<static_cast<unsigned>((n + 255) / 256), 256, 0, stream>>>(
          static_cast<const uint8_t *>(p.src), static_cast<uint8_t *>(p.dst), p.src_plane_stride, p.dst_plane_stride,
          p.src_row_stride, p.dst_row_stride, p.row_bytes, widest_unit(p), p.num_planes, n_out, keep_idx);
    }
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  for (int k = 0; k < n_narrow; ++k) {
    const apack_plane &p = planes[narrow[k]];
    const int64_t n = static_cast<int64_t>(p.num_planes) * n_out;
    const int threads = 256;
    gather_narrow_kernel<<<static_cast<unsigned>((n + threads - 1) / threads), threads, 0, stream>>>(
        static_cast<const uint8_t *>(p.src), static_cast<uint8_t *>(p.dst), p.src_plane_stride, p.dst_plane_stride,
        p.src_row_stride, p.dst_row_stride, p.row_bytes, widest_unit(p), p.num_planes, n_out, keep_idx);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  if (tp.ngroups > 0) {
    static bool attr_done = false;
    if (!attr_done) {
      if (check_cuda(cudaFuncSetAttribute(gather_tma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          kTmaSmem)) != APACK_OK)
        return APACK_ECUDA;
      attr_done = true;
    }
    tp.total_items = static_cast<uint32_t>(items);
    uint64_t blocks = static_cast<uint64_t>(device_sm_count()) * 2;   // two CTAs of kSlots slots per SM
    if (blocks > items) blocks = items;
    gather_tma_kernel<<<static_cast<unsigned>(blocks), 32, kTmaSmem, stream>>>(tp, keep_idx, err);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  if (ip.ngroups > 0) {
    static bool in_attr_done = false;
    if (!in_attr_done) {
      if (check_cuda(cudaFuncSetAttribute(gather_inplace_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                          kInSmem)) != APACK_OK)
        return APACK_ECUDA;
      in_attr_done = true;
    }
    ip.total_items = static_cast<uint32_t>(in_items);
    uint64_t blocks = static_cast<uint64_t>(device_sm_count()) * 2;   // two CTAs per SM, all resident
    if (blocks > kMaxInCtas) blocks = kMaxInCtas;
    if (blocks > in_items) blocks = in_items;
    if (in_items > blocks * 65535) return APACK_EUNSUPPORTED;           // 16-bit progress words
    // the dependency check covers P / gcd(num_planes, P) chunks of every group (at most P <= kInChecks)
    uint32_t period = 1;
    for (int gi = 0; gi < ip.ngroups; ++gi) {
      uint32_t a = ip.g[gi].num_planes, b = static_cast<uint32_t>(blocks);
      while (b) {
        const uint32_t t = a % b;
        a = b;
        b = t;
      }
      const uint32_t per = static_cast<uint32_t>(blocks) / a;
      if (per > period) period = per;
    }
    ip.dep_period = period;
    uint16_t *progress = reinterpret_cast<uint16_t *>(reinterpret_cast<uint8_t *>(err) + kProgressOff);
    if (check_cuda(cudaMemsetAsync(progress, 0, blocks * sizeof(uint16_t), stream)) != APACK_OK) return APACK_ECUDA;
    void *args[] = {&ip, const_cast<int32_t **>(&keep_idx), &progress, &err};
    if (check_cuda(cudaLaunchCooperativeKernel(reinterpret_cast<const void *>(gather_inplace_kernel),
                                               dim3(static_cast<unsigned>(blocks)), dim3(32), args, kInSmem,
                                               stream)) != APACK_OK)
      return APACK_ECUDA;
    count_launches(1);
  }
  return APACK_OK;
}

}  // namespace apack
