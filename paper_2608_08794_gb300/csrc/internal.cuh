// internal.cuh -- declarations shared by the translation units of libapack.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cstddef>
#include <cstdint>

#include "apack.h"

namespace apack {

// Sequences handled by one kernel launch; larger batches take several launches.
constexpr int kSeqsPerLaunch = 64;
// Narrow scoring path: at most this many query rows per KV head group, and in all.
constexpr int kNarrowGroupRows = 32;
constexpr int kNarrowRows = 256;
// Wall-clock limit of every device-side wait.
constexpr uint64_t kWaitLimitNs = 2000000000ull;
// Key splits of the row-statistics pass (upper bound, sizes the workspace).
constexpr int kMaxSplits = 32;

// Device error word at offset 0 of the workspace.
struct DeviceError {
  int32_t code;     // APACK_OK, APACK_ETIMEOUT, APACK_EDEVICE (first error wins)
  int32_t where;    // kernel-specific location code
  int32_t info[2];
};

__device__ __forceinline__ void raise_device_error(DeviceError *e, int32_t code, int32_t where, int32_t a = 0,
                                                   int32_t b = 0) {
  if (atomicCAS(&e->code, 0, code) == 0) {
    e->where = where;
    e->info[0] = a;
    e->info[1] = b;
  }
}

// Workspace carve-up (offsets in bytes from the 256-byte aligned start).
struct WsLayout {
  size_t err_off;     // DeviceError
  size_t part_off;    // float2 [kMaxSplits][sum n_q][Hq]: per-split (max, sum) in log2 units
  size_t lse_off;     // float [qp_rows]: negated log2 normaliser of every packed query row, -inf padding
  size_t qp_off;      // bf16 [qp_rows][128]: query rows repacked per KV head group, 256-row padded
  size_t gsum_off;    // float [Hkv][T]: per head group key sums of the column pass
  size_t mask_off;    // uint32 [key blocks of the batch][8]: which keys of a block count (pass 1)
  // few query rows per head group (narrow path, used instead of the four above):
  bool narrow;
  size_t nlog_off;    // float [sum over sequences of Hq n_q len]: log2-domain logits
  size_t npart_off;   // float2 [sum of Hq n_q ctas]: per-CTA row (max, sum of exp2)
  size_t nlse_off;    // float [sum of Hq n_q]: log2 normalisers
  size_t total;
  int64_t lse_chunks;
  int64_t qp_rows;
};


WsLayout workspace_layout(const apack_seqs *seqs);
int device_sm_count();
void count_launches(uint64_t n);
apack_status check_cuda(cudaError_t e);

// Programmatic dependent launch.  The scoring kernels (both paths) are launched with
// programmatic stream serialization: a kernel may be scheduled while its predecessor on the
// stream drains, and it waits (griddepcontrol.wait, first statement of the kernel) until that
// predecessor has completed and its memory is visible, before any global access.  Each such
// kernel lets its own successor launch early (griddepcontrol.launch_dependents) right after that
// wait.  Measured on GB300, per-step calls: few-row scoring 0.541 -> 0.487 ms summed over the
// paper's 14 steps; the tensor-core scoring chain 0.697 -> 0.675 ms over the 3-step 10-minute
// schedule (a captured graph of the schedule gains nothing: it has no launch gaps to hide).
// Selection and compaction did not gain, so those launch plainly.
__device__ __forceinline__ void pdl_wait_and_release() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t stream,
                       Args &&...args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  at[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}
// Kernel attributes (cudaFuncSetAttribute) belong to the current device: `set` runs once
// per device, recorded in one bit of `done`.  Concurrent first calls on one device may
// both run it, which is harmless (the same attribute is set twice).
template <class F>
cudaError_t once_per_device(std::atomic<uint64_t> &done, F &&set) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const uint64_t bit = (dev >= 0 && dev < 64) ? (uint64_t{1} << dev) : 0;
  if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
  e = set();
  if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_acq_rel);
  return e;
}
bool in_host_memory(const void *p);   // pinned or registered host memory (cudaMemoryTypeHost)

apack_status validate_seqs(const apack_seqs *seqs, int64_t *total_tokens, int64_t *total_qrows);
// Position of sequence b's first query row within the sequence (the causal-row domain's
// rows are tokens q .. q + n_q - 1): q_start_h[b], or len - n_q without q_start_h.
int32_t query_position(const apack_seqs *seqs, int b);

apack_status run_score(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                       float *scores, void *ws, cudaStream_t stream);
bool narrow_score_applies(const apack_seqs *seqs);
void narrow_layout(const apack_seqs *seqs, size_t *logit_floats, size_t *part_float2s, size_t *lse_floats);
apack_status run_score_narrow(const apack_seqs *seqs, const void *q, const void *k, int64_t k_token_stride,
                              float *scores, void *ws, cudaStream_t stream);
apack_status run_select(const apack_seqs *seqs, const float *scores, const int32_t *keep_count_h, int32_t mode,
                        int32_t *keep_idx, uint8_t *modality_out, int32_t *dst_of_src, int32_t *new_cu_seqlens,
                        void *ws, cudaStream_t stream);
// check_only: validate and plan every group, launch nothing (callers that launch other
// kernels first check their compaction this way before any launch).
apack_status run_compact(const int32_t *keep_idx, int64_t n_out, const apack_plane *planes, int32_t num_groups,
                         DeviceError *err, cudaStream_t stream, bool check_only = false);
// 3-D TMA map over a K slab [tokens][hkv][128] bf16 (token_stride bytes between tokens):
// boxes of 64 features x 1 head x box_tokens tokens, 128-byte swizzle.
bool make_kv_tile_map(CUtensorMap *map, const void *k, int hkv, int64_t tokens, int64_t token_stride,
                      uint32_t box_tokens);
apack_status counts_and_offsets(const apack_seqs *s, const float *ratio_h, const int32_t *count_h, int32_t mode,
                                int32_t *k_out, int32_t *cu_out);
bool ws_ok(const apack_seqs *s, const void *ws, size_t bytes);

}  // namespace apack
