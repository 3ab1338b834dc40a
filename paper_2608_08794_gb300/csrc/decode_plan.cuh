// decode_plan.cuh -- launch plan of the decode-step attention, shared by its chunk kernels
// (CUDA-core and tensor-core) and the combine kernel.
#pragma once
#include <cstdint>

#include "internal.cuh"

namespace apack {

struct DecSeq {
  int32_t t0, len;
  int32_t chunk_begin, nchunks;
};

struct DecPlan {
  int32_t nseq, hq, hkv, group, chunk;   // chunk: keys per CTA, a multiple of the kernel's tile
  int32_t total_chunks;
  float scale2;                          // log2(e) / sqrt(128)
  DecSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int find_chunk_seq(const DecPlan &p, int c) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].chunk_begin <= c) ++s;
  return s;
}

// Tensor-core chunk kernel (decode_tc.cu): Hkv = 2 or 4, at most 8 query heads per KV head.
// The CTAs of sequence i claim its 128-key stages from claims[i] (zero before the launch; the
// combine kernel zeroes it again); each writes one partial per query head, in the layout of
// the CUDA-core kernel's chunk partials.
cudaError_t launch_decode_tc(int grid, cudaStream_t stream, const CUtensorMap &kmap, const CUtensorMap &vmap,
                             const DecPlan &P, const uint16_t *q, float *opart, float2 *mlpart, unsigned int *claims,
                             DeviceError *err);

}  // namespace apack
