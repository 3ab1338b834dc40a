// fill.cu -- device twin of synth/gen.py: writes the bf16 draws of stream (seed, tid)
// straight into device memory, bit-identical to the numpy generator
// (SplitMix64 finaliser, Irwin-Hall sum of four 16-bit words, one float32
// multiply, round-to-nearest-even to bf16).  Input generation only.
#include <cuda_runtime.h>

#include <cstdint>

namespace {

__host__ __device__ inline uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

__global__ void fill_normal_bf16_kernel(uint16_t *dst, int64_t n, uint64_t key, uint64_t start, float scale) {
  const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < n; i += stride) {
    const uint64_t h = splitmix64(key ^ splitmix64(start + static_cast<uint64_t>(i)));
    const int64_t s = static_cast<int64_t>((h & 0xFFFFull) + ((h >> 16) & 0xFFFFull) + ((h >> 32) & 0xFFFFull) +
                                           (h >> 48)) - 131070;
    const float z = __fmul_rn(static_cast<float>(s), scale);
    uint32_t b = __float_as_uint(z);
    b = (b + 0x7FFFu + ((b >> 16) & 1u)) >> 16;
    dst[i] = static_cast<uint16_t>(b);
  }
}

}  // namespace

extern "C" {

// n bf16 values of stream (seed, tid), elements start .. start+n-1, into dst.
int synth_fill_normal_bf16(void *dst, int64_t n, uint64_t seed, uint64_t tid, uint64_t start, void *stream) {
  if (n <= 0) return 0;
  const uint64_t key = splitmix64(splitmix64(seed) ^ tid);
  // float32(1 / sqrt((2^32 - 1) / 3)), the constant of synth/gen.py (double sqrt is correctly rounded)
  const double exact = 1.0 / __builtin_sqrt((4294967296.0 - 1.0) / 3.0);
  const float sc = static_cast<float>(exact);
  int64_t blocks = (n + 255) / 256;
  if (blocks > 65536) blocks = 65536;
  fill_normal_bf16_kernel<<<static_cast<unsigned>(blocks), 256, 0, static_cast<cudaStream_t>(stream)>>>(
      static_cast<uint16_t *>(dst), n, key, start, sc);
  return cudaGetLastError() == cudaSuccess ? 0 : 1;
}

}
