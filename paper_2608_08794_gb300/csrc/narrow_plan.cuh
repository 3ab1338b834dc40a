// narrow_plan.cuh -- launch plan of the narrow scoring path, shared by its CUDA-core and
// tensor-core logits kernels and by the merge and final kernels.
#pragma once
#include <cstdint>

#include "internal.cuh"

namespace apack {

struct NSeq {
  int32_t t0, len;
  int32_t q_off, n_q;
  int32_t unit_begin;                  // first 256-key CTA of this sequence (general logits, final)
  int32_t unit8_begin;                 // first chunk (CTA) of this sequence in the rows8 logits kernel
  int32_t nparts;                      // CTA partials of the logits kernel in use
  int32_t rows;                        // logit rows R = Hq * n_q
  int32_t q_pos;                       // causal rows: position of query row 0 within the sequence
  int64_t lstride;                     // logit row stride: len rounded up to kLogitPad
  int64_t logit_base;                  // float offset of this sequence's logits [R][lstride]
  int64_t part_base;                   // float2 offset of its CTA partials [nparts][R]
  int64_t lse_base;                    // float offset of its lse2 [R]
};

struct NarrowPlan {
  int32_t nseq;
  int32_t total_units;
  int32_t total_units8;
  int32_t chunk;                       // keys per CTA of the rows8 kernel (a multiple of the kernel's tile)
  int32_t hq, hkv, group;
  int32_t causal;                      // APACK_SOFTMAX_CAUSAL_ROW: row r of n_q sees keys <= q_pos + r
  float scale2;
  NSeq seq[kSeqsPerLaunch];
};

__device__ __forceinline__ int find_unit_seq(const NarrowPlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit_begin <= u) ++s;
  return s;
}

__device__ __forceinline__ int find_unit8_seq(const NarrowPlan &p, int u) {
  int s = 0;
  while (s + 1 < p.nseq && p.seq[s + 1].unit8_begin <= u) ++s;
  return s;
}

// Tensor-core logits kernel of the narrow path (score_narrow_tc.cu): Hkv = 2 or 4, at most 8
// query rows per KV head group, chunks of P.chunk keys (a multiple of 128) per CTA.
cudaError_t launch_narrow_tc(int grid, cudaStream_t stream, const CUtensorMap &kmap, const NarrowPlan &P,
                             const uint16_t *q, const uint8_t *modality, float *logits, float2 *part,
                             DeviceError *err);

}  // namespace apack
