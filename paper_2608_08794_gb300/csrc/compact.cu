// compact.cu -- KV-cache and hidden-state slicing of Sec. 3.2 (Algorithm 1, "slice their
// KV-cache entries"): dst row j = src row keep_idx[j] for every plane.
//
// This file plans a call (validating every group before anything is launched) and holds the
// small paths; the bulk paths live beside it:
//  - rows of 16-byte multiples up to 32 KB, 16-byte aligned, out of place: the bulk-copy (TMA)
//    gather of compact_tma.cu;
//  - the same rows in place (src == dst): compact_inplace.cu;
//  - a source in pinned host memory: the zero-copy gather below;
//  - rows that are not 16-byte multiples (or misaligned): the narrow kernel below, one thread
//    per row.
#include "compact_plan.cuh"

namespace apack {

using namespace gather;

namespace {

// ------------------------------------------------------------------ host source
// Source rows in pinned host memory (zero copy): only the kept rows cross the host link.
// Consecutive threads take consecutive 16-byte pieces of a row (coalesced link reads); each
// thread issues U loads before its U stores so that enough reads are in flight.  Every CTA moves
// a fixed 64 KB and exits (no grid-stride loop): CTAs of kernels on other streams (scoring and
// selection beside a link-bound gather) then get SMs as soon as gather CTAs retire, first when
// their stream has the higher priority.
constexpr int kHostUnroll = 4;
constexpr int kHostRounds = 4;
constexpr int64_t kHostPiecesPerCta = 256 * kHostUnroll * kHostRounds;   // 16-byte pieces

__global__ void __launch_bounds__(256) gather_host_kernel(const uint8_t *__restrict__ src, uint8_t *__restrict__ dst,
                                                          int64_t sps, int64_t dps, int64_t srs, int64_t drs,
                                                          int64_t row_bytes, int64_t n_planes, int64_t n_out,
                                                          const int32_t *__restrict__ keep_idx) {
  const int64_t vec_per_row = row_bytes / 16;
  const int64_t total = n_planes * n_out * vec_per_row;
  const int64_t cta0 = static_cast<int64_t>(blockIdx.x) * kHostPiecesPerCta + threadIdx.x;
#pragma unroll 1
  for (int r = 0; r < kHostRounds; ++r) {
    const int64_t base = cta0 + r * (256 * kHostUnroll);
    uint4 v[kHostUnroll];
#pragma unroll
    for (int u = 0; u < kHostUnroll; ++u) {
      const int64_t e = base + u * 256;
      if (e < total) {
        const int64_t row = e / vec_per_row, c = e - row * vec_per_row;
        const int64_t plane = row / n_out, j = row - plane * n_out;
        v[u] = *reinterpret_cast<const uint4 *>(src + plane * sps + static_cast<int64_t>(keep_idx[j]) * srs + c * 16);
      }
    }
#pragma unroll
    for (int u = 0; u < kHostUnroll; ++u) {
      const int64_t e = base + u * 256;
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
                         DeviceError *err, cudaStream_t stream, bool check_only) {
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
      if (widest_unit(p) == 16 && static_cast<int64_t>(p.num_planes) * n_out * (p.row_bytes / 16) >
                                      0x7FFFFFFFLL * kHostPiecesPerCta)
        return APACK_EUNSUPPORTED;                  // beyond one launch's grid
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
  uint32_t in_blocks = 0;
  if (ip.ngroups > 0) {
    const apack_status st = plan_inplace(ip, in_items, &in_blocks);
    if (st != APACK_OK) return st;
  }
  if (check_only) return APACK_OK;
  for (int k = 0; k < n_host; ++k) {
    const apack_plane &p = host_groups[k];
    if (widest_unit(p) == 16) {
      const int64_t n = static_cast<int64_t>(p.num_planes) * n_out * (p.row_bytes / 16);
      const int64_t blocks = (n + kHostPiecesPerCta - 1) / kHostPiecesPerCta;   // checked when planned
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
    tp.total_items = static_cast<uint32_t>(items);
    if (launch_out_of_place(tp, keep_idx, err, stream) != APACK_OK) return APACK_ECUDA;
  }
  if (ip.ngroups > 0 && launch_inplace(ip, in_blocks, keep_idx, err, stream) != APACK_OK) return APACK_ECUDA;
  return APACK_OK;
}

}  // namespace apack
