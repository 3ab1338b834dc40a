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
  uint32_t pad;
};

struct TmaPlan {
  int32_t ngroups;
  uint32_t total_items;
  uint32_t n_out;
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
  it.plane = local / G.chunks_per_plane;
  it.r0 = (local - it.plane * G.chunks_per_plane) * G.rows_per_slot;
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
  for (uint32_t j = 0; j < n_mine && j < kSlots; ++j)
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
    }
  }
  if (!ok) {
    // loads of items j .. j+kSlots-1 may still be in flight: wait for them (bounded)
    for (uint32_t k = j; k < n_mine && k < j + kSlots; ++k) mbar_wait(&full[k % kSlots], (k / kSlots) & 1u, kWaitLimitNs / 4);
  }
  bulk_wait_all();
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
  TmaPlan tp{};
  tp.n_out = static_cast<uint32_t>(n_out);
  uint64_t items = 0;
  int narrow[kMaxGroups * 4];
  int n_narrow = 0;
  for (int i = 0; i < num_groups; ++i) {
    const apack_plane &p = planes[i];
    if (p.num_planes < 0 || p.row_bytes < 0) return APACK_EINVAL;
    if (p.num_planes == 0 || p.row_bytes == 0) continue;
    if (!p.src || !p.dst || p.src_row_stride < p.row_bytes || p.dst_row_stride < p.row_bytes ||
        p.src_plane_stride < 0 || p.dst_plane_stride < 0)
      return APACK_EINVAL;
    if (p.src == p.dst) return APACK_EUNSUPPORTED;   // in-place compaction is not offered by this build
    if (ranges_overlap(p, n_out, n_out)) return APACK_EINVAL;
    if (widest_unit(p) == 16 && p.row_bytes <= static_cast<int64_t>(kSlotBytes)) {
      if (tp.ngroups == kMaxGroups) return APACK_EINVAL;
      TmaGroup &g = tp.g[tp.ngroups++];
      g.src = static_cast<const uint8_t *>(p.src);
      g.dst = static_cast<uint8_t *>(p.dst);
      g.sps = p.src_plane_stride;
      g.dps = p.dst_plane_stride;
      g.srs = p.src_row_stride;
      g.drs = p.dst_row_stride;
      g.row_bytes = static_cast<uint32_t>(p.row_bytes);
      g.rows_per_slot = kSlotBytes / g.row_bytes;
      g.chunks_per_plane = static_cast<uint32_t>((n_out + g.rows_per_slot - 1) / g.rows_per_slot);
      g.item_begin = static_cast<uint32_t>(items);
      g.contiguous = p.dst_row_stride == p.row_bytes;
      items += static_cast<uint64_t>(g.chunks_per_plane) * p.num_planes;
      if (items > 0x7FFFFFFFull) return APACK_EINVAL;
    } else {
      if (n_narrow == kMaxGroups * 4) return APACK_EINVAL;
      narrow[n_narrow++] = i;
    }
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
  return APACK_OK;
}

}  // namespace apack
