// compact.cu -- KV-cache and hidden-state slicing of Sec. 3.2 (Algorithm 1, "slice their
// KV-cache entries"): dst row j = src row keep_idx[j] for every plane.
//
// HBM-bound: every byte is read once and written once.  The wide kernel moves
// rows in 512-byte pieces (one 16-byte vector per lane of a warp), with
// kUnroll pieces in flight per warp before any store; loads bypass L1 and
// stores are marked streaming so that the copy does not evict the L2 working
// set.  Rows that are not 16-byte multiples (or misaligned) take the narrow
// kernel, one thread per row.
#include "internal.cuh"

namespace apack {

namespace {

constexpr int kMaxGroups = 16;
constexpr int kWideThreads = 256;
constexpr int kUnroll = 4;

struct WideGroup {
  const uint8_t *src;
  uint8_t *dst;
  int64_t sps, dps, srs, drs;   // plane and row strides in bytes
  uint32_t vecs;                // 16-byte vectors per row
  uint32_t pieces;              // 512-byte pieces per row = ceil(vecs / 32)
  uint32_t n_planes;
  uint32_t item_begin;          // first piece index of this group
};

struct WidePlan {
  int32_t ngroups;
  uint32_t total_items;
  uint32_t n_out;
  WideGroup g[kMaxGroups];
};

__device__ __forceinline__ uint4 ld_stream(const void *p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ void st_stream(void *p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
               : "memory");
}

__global__ void __launch_bounds__(kWideThreads)
    gather_wide_kernel(const __grid_constant__ WidePlan plan, const int32_t *__restrict__ keep_idx) {
  const int lane = threadIdx.x & 31;
  const uint32_t warp = (blockIdx.x * kWideThreads + threadIdx.x) >> 5;
  const uint32_t nwarps = (gridDim.x * kWideThreads) >> 5;
  for (uint32_t batch = warp; batch * kUnroll < plan.total_items; batch += nwarps) {
    uint4 v[kUnroll];
    uint8_t *dptr[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      dptr[u] = nullptr;
      const uint32_t item = batch * kUnroll + u;
      if (item >= plan.total_items) continue;
      int gi = 0;
      while (gi + 1 < plan.ngroups && plan.g[gi + 1].item_begin <= item) ++gi;
      const WideGroup &G = plan.g[gi];
      const uint32_t local = item - G.item_begin;
      const uint32_t rowplane = local / G.pieces;
      const uint32_t piece = local - rowplane * G.pieces;
      const uint32_t plane = rowplane / plan.n_out;
      const uint32_t row = rowplane - plane * plan.n_out;
      const uint32_t vec = piece * 32 + lane;
      if (vec >= G.vecs) continue;
      const int64_t src_row = keep_idx[row];
      v[u] = ld_stream(G.src + plane * G.sps + src_row * G.srs + vec * 16ull);
      dptr[u] = G.dst + plane * G.dps + static_cast<int64_t>(row) * G.drs + vec * 16ull;
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u)
      if (dptr[u]) st_stream(dptr[u], v[u]);
  }
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
                         cudaStream_t stream) {
  if (n_out < 0 || num_groups < 0 || (num_groups > 0 && !planes)) return APACK_EINVAL;
  if (n_out == 0 || num_groups == 0) return APACK_OK;
  if (!keep_idx || n_out > INT32_MAX) return APACK_EINVAL;
  WidePlan wp{};
  wp.n_out = static_cast<uint32_t>(n_out);
  uint64_t items = 0;
  const int sms = device_sm_count();
  for (int i = 0; i < num_groups; ++i) {
    const apack_plane &p = planes[i];
    if (p.num_planes < 0 || p.row_bytes < 0) return APACK_EINVAL;
    if (p.num_planes == 0 || p.row_bytes == 0) continue;
    if (!p.src || !p.dst || p.src_row_stride < p.row_bytes || p.dst_row_stride < p.row_bytes ||
        p.src_plane_stride < 0 || p.dst_plane_stride < 0)
      return APACK_EINVAL;
    if (p.src == p.dst) return APACK_EUNSUPPORTED;   // in-place compaction is not offered by this build
    if (ranges_overlap(p, n_out, n_out)) return APACK_EINVAL;
    const int unit = widest_unit(p);
    if (unit == 16 && p.row_bytes >= 256) {
      if (wp.ngroups == kMaxGroups) return APACK_EINVAL;
      WideGroup &g = wp.g[wp.ngroups++];
      g.src = static_cast<const uint8_t *>(p.src);
      g.dst = static_cast<uint8_t *>(p.dst);
      g.sps = p.src_plane_stride;
      g.dps = p.dst_plane_stride;
      g.srs = p.src_row_stride;
      g.drs = p.dst_row_stride;
      g.vecs = static_cast<uint32_t>(p.row_bytes / 16);
      g.pieces = (g.vecs + 31) / 32;
      g.n_planes = static_cast<uint32_t>(p.num_planes);
      g.item_begin = static_cast<uint32_t>(items);
      items += static_cast<uint64_t>(g.pieces) * p.num_planes * static_cast<uint64_t>(n_out);
      if (items > 0x7FFFFFFFull) return APACK_EINVAL;
    } else {
      const int64_t n = static_cast<int64_t>(p.num_planes) * n_out;
      const int threads = 256;
      gather_narrow_kernel<<<static_cast<unsigned>((n + threads - 1) / threads), threads, 0, stream>>>(
          static_cast<const uint8_t *>(p.src), static_cast<uint8_t *>(p.dst), p.src_plane_stride,
          p.dst_plane_stride, p.src_row_stride, p.dst_row_stride, p.row_bytes, unit, p.num_planes, n_out, keep_idx);
      count_launches(1);
      if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
    }
  }
  if (wp.ngroups > 0) {
    wp.total_items = static_cast<uint32_t>(items);
    const uint64_t batches = (items + kUnroll - 1) / kUnroll;
    const uint64_t warps_per_block = kWideThreads / 32;
    uint64_t blocks = (batches + warps_per_block - 1) / warps_per_block;
    const uint64_t cap = static_cast<uint64_t>(sms) * 8;   // 8 resident blocks of 256 threads per SM
    if (blocks > cap) blocks = cap;
    gather_wide_kernel<<<static_cast<unsigned>(blocks), kWideThreads, 0, stream>>>(wp, keep_idx);
    count_launches(1);
    if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  }
  return APACK_OK;
}

}  // namespace apack
