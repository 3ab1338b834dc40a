// compact_plan.cuh -- the item plan shared by the bulk-copy gathers of Sec. 3.2's slicing step
// (Algorithm 1, "slice their KV-cache entries"): compact.cu (out of place) and compact_inplace.cu
// (in place).  An item is one 32 KB shared-memory slot's worth of kept rows of one plane.
#pragma once
#include "internal.cuh"
#include "ptx.cuh"

namespace apack {
namespace gather {

constexpr int kMaxGroups = 16;
constexpr uint32_t kSlotBytes = 32768;

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

// Out of place (compact_tma.cu): tp.total_items set, at least one item.
apack_status launch_out_of_place(const TmaPlan &tp, const int32_t *keep_idx, DeviceError *err,
                                 cudaStream_t stream);

// In place (compact_inplace.cu).  plan_inplace sizes the cooperative launch (APACK_EUNSUPPORTED
// when the items exceed what 16-bit progress words count); launch_inplace zeroes the progress
// words in the workspace (bytes 256..1023 past err) and launches.
apack_status plan_inplace(TmaPlan &ip, uint64_t in_items, uint32_t *blocks);
apack_status launch_inplace(const TmaPlan &ip, uint32_t blocks, const int32_t *keep_idx, DeviceError *err,
                            cudaStream_t stream);

}  // namespace gather
}  // namespace apack
