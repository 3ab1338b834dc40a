// compact_tma.cu -- out-of-place slicing for Sec. 3.2's compaction step (Algorithm 1, "slice their
// KV-cache entries"): dst row j = src row keep_idx[j] of every plane, for rows of 16-byte multiples
// up to 32 KB, 16-byte aligned.
//
// HBM-bound: every byte is read once and written once.  Each copy warp streams kept rows into a
// ring of 32 KB shared-memory slots with cp.async.bulk (one row per lane, completion on the slot's
// mbarrier) and writes each slot back with a single bulk store when the output rows are
// contiguous (one per row otherwise).  Two slots per warp and three independent copy warps per
// CTA, one CTA per SM (192 KB in flight per SM).  Measured on the 48-plane first 10-minute step:
// 0.854 ms, against 0.858-0.863 ms for the same warps as three one-warp CTAs per SM, 0.932-0.939
// ms with three slots in each of two one-warp CTAs (the same bytes in flight, fewer warps issuing
// copies) and 1.18 ms with seven slots in one; 16 KB or 24 KB slots in more CTAs were slower too.
// On fewer SMs the rate falls (128 SMs: 0.886 ms, 96: 1.076 ms): one SM moves about 50 GB/s.
#include "compact_plan.cuh"

namespace apack {
namespace gather {
namespace {

constexpr int kSlots = 2;                       // slots per copy warp
constexpr uint32_t kTmaSmem = kSlots * kSlotBytes;  // per copy warp

constexpr int kWarps = 3;                       // independent copy warps per CTA
__global__ void __launch_bounds__(32 * kWarps) gather_tma_kernel(const __grid_constant__ TmaPlan plan,
                                                                 const int32_t *__restrict__ keep_idx, DeviceError *err) {
  extern __shared__ __align__(1024) uint8_t smem_all[];
  __shared__ __align__(8) uint64_t full_all[kWarps][kSlots];
  pdl_wait_and_release();   // keep_idx and the source rows are complete; the next launch may be scheduled
  const int lane = threadIdx.x & 31, wv = threadIdx.x >> 5;
  uint8_t *slots = smem_all + wv * kTmaSmem;
  uint64_t *full = full_all[wv];
  if (lane == 0) {
    for (int i = 0; i < kSlots; ++i) mbar_init(&full[i], 1);
    fence_mbar_init();
  }
  __syncwarp();
  // this warp's items: w, w + W, w + 2W, ... for copy warp w of the W in the grid
  const uint32_t first = blockIdx.x * kWarps + wv, stride = gridDim.x * kWarps;
  const uint32_t n_mine = first < plan.total_items ? (plan.total_items - first + stride - 1) / stride : 0;
  uint32_t issued = n_mine < kSlots ? n_mine : kSlots;
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

}  // namespace

apack_status launch_out_of_place(const TmaPlan &tp, const int32_t *keep_idx, DeviceError *err,
                                 cudaStream_t stream) {
  static std::atomic<uint64_t> attr_done{0};
  if (once_per_device(attr_done, [] {
        return cudaFuncSetAttribute(gather_tma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kTmaSmem * kWarps);
      }) != cudaSuccess)
    return APACK_ECUDA;
  uint64_t blocks = static_cast<uint64_t>(device_sm_count());   // one CTA per SM
  if (blocks * kWarps > tp.total_items) blocks = (tp.total_items + kWarps - 1) / kWarps;
  const cudaError_t e = launch_pdl(gather_tma_kernel, dim3(static_cast<unsigned>(blocks)), dim3(32 * kWarps),
                                   kTmaSmem * kWarps, stream, tp, keep_idx, err);
  count_launches(1);
  return check_cuda(e);
}

}  // namespace gather
}  // namespace apack
