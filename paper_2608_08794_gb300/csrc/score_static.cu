// score_static.cu -- apack_score_static: the relevance scores of apack_score for callers
// that cannot allocate device memory.
//
// Who needs it: a plugin running inside an inference engine that owns every device
// allocation (the plugin gets its input and output tensors but may not call
// cudaMalloc), or a serving process that fixes its device memory when it starts so
// that no request can fail on an out-of-memory allocation later.  Such a caller has
// no way to provide the scratch workspace apack_score needs.
//
// Here the scratch is one file-scope device array of kStaticScratchBytes, reserved
// on every GPU that loads this library for as long as the process lives.  The host
// code looks up its device address once per device (cudaGetSymbolAddress, with that
// device current) on the first call made on that device, and passes it to the same
// scoring kernels apack_score launches.  No call allocates, frees or calls an
// allocating library routine.
#include <atomic>

#include "internal.cuh"

namespace {

constexpr size_t kStaticScratchBytes = static_cast<size_t>(8) << 20;   // 8 MiB
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_score_scratch[kStaticScratchBytes];

std::atomic<void *> g_scratch_addr[kMaxDevices];

}  // namespace

extern "C" apack_status apack_score_static(const apack_seqs *seqs, const void *q, const void *k,
                                           int64_t k_token_stride, float *scores, int32_t *device_error_out,
                                           void *stream) {
  using namespace apack;
  int64_t T = 0, NQ = 0;
  apack_status st = validate_seqs(seqs, &T, &NQ);
  if (st != APACK_OK) return st;
  // Pointer checks come before any device work, as in apack_score: q and k are
  // read by TMA, so they must be device memory.
  if (!q || !k || !scores) return APACK_EINVAL;
  if (in_host_memory(k) || in_host_memory(q)) return APACK_EINVAL;
  // The whole scratch of the batch must fit the fixed array.
  if (workspace_layout(seqs).total > kStaticScratchBytes) return APACK_EWORKSPACE;
  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return APACK_ECUDA;
  if (dev < 0 || dev >= kMaxDevices) return APACK_EUNSUPPORTED;
  void *ws = g_scratch_addr[dev].load(std::memory_order_acquire);
  if (!ws) {
    // First call on this device: the array's device address (a host-side name of
    // the array is not a device address).
    if (cudaGetSymbolAddress(&ws, g_score_scratch) != cudaSuccess || !ws) return APACK_ECUDA;
    g_scratch_addr[dev].store(ws, std::memory_order_release);
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // The array keeps whatever the previous call left; only the error word has to
  // start at zero (every other region is written before it is read).
  if (cudaMemsetAsync(ws, 0, sizeof(DeviceError), s) != cudaSuccess) return APACK_ECUDA;
  st = run_score(seqs, q, k, k_token_stride, scores, ws, s);
  if (st != APACK_OK) return st;
  if (device_error_out &&
      cudaMemcpyAsync(device_error_out, ws, sizeof(int32_t), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
    return APACK_ECUDA;
  return APACK_OK;
}
