// prellm.cu -- pre-LLM frame alignment of A-PACK (Sec. 3.1, "Coarse pass" and "Gated fine
// pass"; Eq. cka and Eq. gate; Algorithm 1, the first steps of the pre-LLM stage).
//
//  pool kernel:  v_f = mean of frame f's visual tokens, a_f = mean of the audio tokens
//                resampled onto frame f (token j -> frame floor(j F / N_a)); fp32 sums
//                of bf16 rows in token order.  Reads every encoder token once: the
//                HBM-bound part of this stage.
//  cka kernel:   one CTA per frame; over the window W_f (cut to the clip) the rows are
//                centred and the w x w Grams K_A = A A^T, K_V = V V^T accumulated over
//                the feature dimension, which gives Eq. cka exactly since
//                ||V^T A||_F^2 = <K_A, K_V>_F and ||A^T A||_F = ||K_A||_F; also the
//                direct distance d_f = ||v_f - a_f||.
//  gate:         the last CTA of the CKA kernel to finish (a counter in the workspace,
//                zeroed by the pool kernel) computes c-bar, min/max of d, the min-max
//                normalised distance and the gated score s_f of Eq. gate (blend when
//                c-bar < tau) over the whole clip.
// All reductions run in a fixed order: results are deterministic.  Two launches per call; the
// CKA kernel is a programmatic dependent of the pool kernel (scheduled while the pool drains,
// waiting for its completion before any read).
#include <algorithm>
#include <cmath>

#include "internal.cuh"

namespace apack {

namespace {

constexpr int kPoolMaxThreads = 512;   // 8 features per thread: up to 4096 features per CTA
constexpr int kCkaThreads = 256;
constexpr int kMaxWindow = 7;

__device__ __forceinline__ void add_bf16x8(const uint4 &v, float (&acc)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    acc[2 * i] += __uint_as_float(w[i] << 16);
    acc[2 * i + 1] += __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__global__ void __launch_bounds__(kPoolMaxThreads, 2)
    frame_pool_kernel(const uint4 *__restrict__ visual, const uint4 *__restrict__ audio, int n_frames, int tpf,
                      int n_audio, int64_t dim, float *__restrict__ v_out, float *__restrict__ a_out,
                      unsigned int *done) {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");   // the CKA kernel may be scheduled
  const int f = blockIdx.x;
  if (f == 0 && blockIdx.y == 0 && threadIdx.x == 0) *done = 0u;   // CTA counter of the CKA kernel
  const int64_t fi = (static_cast<int64_t>(blockIdx.y) * blockDim.x + threadIdx.x) * 8;
  if (fi >= dim) return;
  const int64_t vec_per_row = dim / 8;
  const int64_t col = fi / 8;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  const int64_t r0 = static_cast<int64_t>(f) * tpf;
#pragma unroll 8
  for (int t = 0; t < tpf; ++t) add_bf16x8(__ldg(visual + (r0 + t) * vec_per_row + col), acc);
  const float inv_v = 1.f / static_cast<float>(tpf);
#pragma unroll
  for (int i = 0; i < 8; ++i) v_out[static_cast<int64_t>(f) * dim + fi + i] = acc[i] * inv_v;
  // audio tokens j with floor(j F / N_a) == f: j in [ceil(f N_a / F), ceil((f+1) N_a / F))
  const int64_t j0 = (static_cast<int64_t>(f) * n_audio + n_frames - 1) / n_frames;
  const int64_t j1 = (static_cast<int64_t>(f + 1) * n_audio + n_frames - 1) / n_frames;
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.f;
#pragma unroll 8
  for (int64_t j = j0; j < j1; ++j) add_bf16x8(__ldg(audio + j * vec_per_row + col), acc);
  const float inv_a = 1.f / static_cast<float>(j1 - j0);
#pragma unroll
  for (int i = 0; i < 8; ++i) a_out[static_cast<int64_t>(f) * dim + fi + i] = acc[i] * inv_a;
}

// Per-frame windowed CKA (Eq. cka) and direct distance; the last CTA to finish also
// runs the gate (Eq. gate) over all frames.  W is the window size (odd, <= kMaxWindow);
// windows cut by the clip's ends hold w < W rows and the missing rows are zeros that
// never enter a Gram entry with i or j >= w.
template <int W>
__global__ void __launch_bounds__(kCkaThreads)
    frame_cka_gate_kernel(const float *__restrict__ v, const float *__restrict__ a, int n_frames, int64_t dim,
                          float tau, float beta, unsigned int *done, float *__restrict__ c_out,
                          float *__restrict__ d_out, float *__restrict__ s_out, float *__restrict__ dn_out,
                          float *__restrict__ cbar_out) {
  pdl_wait_and_release();   // the pooled rows (and the zeroed counter) of the pool kernel are visible
  constexpr int kG = W * (W + 1) / 2;
  constexpr int kN = 2 * kG + 1;
  constexpr int kWarps = kCkaThreads / 32;
  __shared__ float red[kWarps][kN];
  __shared__ float tot[kN];
  __shared__ bool last;
  const int f = blockIdx.x;
  const int lo = max(0, f - W / 2), hi = min(n_frames, f + W / 2 + 1);
  const int w = hi - lo;
  const int center = f - lo;
  const float inv_w = 1.f / static_cast<float>(w);
  float ga[kG], gv[kG], dist = 0.f;
#pragma unroll
  for (int i = 0; i < kG; ++i) ga[i] = gv[i] = 0.f;
  // four consecutive features per thread and step (16-byte loads of the pooled rows: dim is a
  // multiple of 8 and the rows start 256-byte aligned)
  const int64_t nv4 = dim / 4;
  const float4 *a4 = reinterpret_cast<const float4 *>(a);
  const float4 *v4 = reinterpret_cast<const float4 *>(v);
  for (int64_t x = threadIdx.x; x < nv4; x += kCkaThreads) {
    float4 a_r[W], v_r[W];
#pragma unroll
    for (int r = 0; r < W; ++r) {
      a_r[r] = r < w ? a4[static_cast<int64_t>(lo + r) * nv4 + x] : make_float4(0.f, 0.f, 0.f, 0.f);
      v_r[r] = r < w ? v4[static_cast<int64_t>(lo + r) * nv4 + x] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int e = 0; e < 4; ++e) {             // the four features in order
      float av[W], vv[W], am = 0.f, vm = 0.f, dd = 0.f;
#pragma unroll
      for (int r = 0; r < W; ++r) {
        av[r] = e == 0 ? a_r[r].x : e == 1 ? a_r[r].y : e == 2 ? a_r[r].z : a_r[r].w;
        vv[r] = e == 0 ? v_r[r].x : e == 1 ? v_r[r].y : e == 2 ? v_r[r].z : v_r[r].w;
        am += av[r];
        vm += vv[r];
        if (r == center) dd = vv[r] - av[r];
      }
      dist = fmaf(dd, dd, dist);
      am *= inv_w;
      vm *= inv_w;
#pragma unroll
      for (int r = 0; r < W; ++r) {
        av[r] = r < w ? av[r] - am : 0.f;
        vv[r] = r < w ? vv[r] - vm : 0.f;
      }
      int k = 0;
#pragma unroll
      for (int i = 0; i < W; ++i)
#pragma unroll
        for (int j = i; j < W; ++j, ++k) {
          ga[k] = fmaf(av[i], av[j], ga[k]);
          gv[k] = fmaf(vv[i], vv[j], gv[k]);
        }
    }
  }
  // fixed-order block reduction: warp trees, then one thread per sum over the warps in order
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int i = 0; i < kG; ++i) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      ga[i] += __shfl_xor_sync(0xffffffffu, ga[i], o);
      gv[i] += __shfl_xor_sync(0xffffffffu, gv[i], o);
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) dist += __shfl_xor_sync(0xffffffffu, dist, o);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kG; ++i) {
      red[warp][i] = ga[i];
      red[warp][kG + i] = gv[i];
    }
    red[warp][2 * kG] = dist;
  }
  __syncthreads();
  if (threadIdx.x < kN) {
    float t = 0.f;
#pragma unroll
    for (int wp = 0; wp < kWarps; ++wp) t += red[wp][threadIdx.x];
    tot[threadIdx.x] = t;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    // <K_A, K_V>_F, ||K_A||_F^2 and ||K_V||_F^2 from the upper triangles (off-diagonal entries twice)
    float dot = 0.f, na = 0.f, nv = 0.f;
    int k = 0;
#pragma unroll
    for (int i = 0; i < W; ++i)
#pragma unroll
      for (int j = i; j < W; ++j, ++k) {
        const float m = (i == j) ? 1.f : 2.f;
        dot = fmaf(m * tot[k], tot[kG + k], dot);
        na = fmaf(m * tot[k], tot[k], na);
        nv = fmaf(m * tot[kG + k], tot[kG + k], nv);
      }
    const float den = sqrtf(na) * sqrtf(nv);
    c_out[f] = den > 0.f ? dot / den : 0.f;
    d_out[f] = sqrtf(tot[2 * kG]);
    __threadfence();
    last = atomicAdd(done, 1u) == static_cast<unsigned>(n_frames - 1);
  }
  __syncthreads();
  if (!last) return;
  // gate over the whole clip (every other CTA's c and d are visible after its fence)
  __threadfence();
  __shared__ double rsum[kWarps];
  __shared__ float rmin[kWarps], rmax[kWarps];
  __shared__ double cbar_s;
  __shared__ float dmin_s, dmax_s;
  const volatile float *cv = c_out;
  const volatile float *dv = d_out;
  double cs = 0.0;
  float mn = INFINITY, mx = -INFINITY;
  for (int g = threadIdx.x; g < n_frames; g += kCkaThreads) {
    cs += cv[g];
    const float dg = dv[g];
    mn = fminf(mn, dg);
    mx = fmaxf(mx, dg);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    cs += __shfl_xor_sync(0xffffffffu, cs, o);
    mn = fminf(mn, __shfl_xor_sync(0xffffffffu, mn, o));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  }
  if (lane == 0) {
    rsum[warp] = cs;
    rmin[warp] = mn;
    rmax[warp] = mx;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t = 0.0;
    float lo_d = INFINITY, hi_d = -INFINITY;
    for (int wp = 0; wp < kWarps; ++wp) {
      t += rsum[wp];
      lo_d = fminf(lo_d, rmin[wp]);
      hi_d = fmaxf(hi_d, rmax[wp]);
    }
    cbar_s = t / n_frames;
    dmin_s = lo_d;
    dmax_s = hi_d;
    if (cbar_out) *cbar_out = static_cast<float>(cbar_s);
  }
  __syncthreads();
  const bool blend = cbar_s < static_cast<double>(tau);
  const float span = dmax_s - dmin_s;
  for (int g = threadIdx.x; g < n_frames; g += kCkaThreads) {
    const float cg = cv[g];
    const float dn = span > 0.f ? (dv[g] - dmin_s) / span : 0.f;
    if (dn_out) dn_out[g] = dn;
    s_out[g] = blend ? (1.f - beta) * cg + beta * (1.f - dn) : cg;
  }
}

size_t up(size_t x) { return (x + 255) & ~static_cast<size_t>(255); }

}  // namespace

}  // namespace apack

using namespace apack;

extern "C" {

apack_status apack_frame_alignment_workspace_size(int32_t n_frames, int64_t dim, size_t *bytes) {
  if (!bytes || n_frames < 1 || dim < 8) return APACK_EINVAL;
  // error word, v [F][dim], a [F][dim], c [F], d [F], scratch
  *bytes = 256 + 2 * up(static_cast<size_t>(n_frames) * dim * sizeof(float)) +
           2 * up(static_cast<size_t>(n_frames) * sizeof(float)) + 256;
  return APACK_OK;
}

apack_status apack_frame_alignment(const void *visual, const void *audio, int32_t n_frames, int32_t tokens_per_frame,
                                   int32_t n_audio, int64_t dim, int32_t window, float tau, float beta, float *c_out,
                                   float *s_out, float *dnorm_out, float *cbar_out, void *ws, size_t ws_bytes,
                                   void *stream) {
  if (!visual || !audio || !c_out || !s_out || !ws) return APACK_EINVAL;
  if (n_frames < 1 || tokens_per_frame < 1 || n_audio < n_frames || dim < 8 || (dim % 8) != 0) return APACK_EINVAL;
  if (window < 1 || window > kMaxWindow || (window % 2) == 0) return APACK_EINVAL;
  if (!(beta >= 0.f && beta <= 1.f) || !std::isfinite(tau)) return APACK_EINVAL;
  if ((reinterpret_cast<uintptr_t>(visual) & 15) || (reinterpret_cast<uintptr_t>(audio) & 15) ||
      (reinterpret_cast<uintptr_t>(ws) & 255))
    return APACK_EINVAL;
  size_t need = 0;
  apack_frame_alignment_workspace_size(n_frames, dim, &need);
  if (ws_bytes < need) return APACK_EWORKSPACE;
  uint8_t *w = static_cast<uint8_t *>(ws);
  unsigned int *done = reinterpret_cast<unsigned int *>(w);
  float *vbuf = reinterpret_cast<float *>(w + 256);
  float *abuf = reinterpret_cast<float *>(w + 256 + up(static_cast<size_t>(n_frames) * dim * sizeof(float)));
  float *dbuf = reinterpret_cast<float *>(w + 256 + 2 * up(static_cast<size_t>(n_frames) * dim * sizeof(float)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // one CTA per frame covers up to 4096 features; wider rows take more CTAs per frame
  const int64_t vecs = dim / 8;
  const int pthreads = static_cast<int>(std::min<int64_t>(kPoolMaxThreads, (vecs + 31) / 32 * 32));
  dim3 pgrid(n_frames, static_cast<unsigned>((vecs + pthreads - 1) / pthreads));
  frame_pool_kernel<<<pgrid, pthreads, 0, s>>>(static_cast<const uint4 *>(visual), static_cast<const uint4 *>(audio),
                                              n_frames, tokens_per_frame, n_audio, dim, vbuf, abuf, done);
  count_launches(1);
  if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  // programmatic dependent launch: the CKA kernel's CTAs are scheduled while the pool kernel drains
  cudaError_t e = cudaSuccess;
  switch (window) {
    case 1:
      e = launch_pdl(frame_cka_gate_kernel<1>, dim3(n_frames), dim3(kCkaThreads), 0, s, vbuf, abuf, n_frames, dim,
                     tau, beta, done, c_out, dbuf, s_out, dnorm_out, cbar_out);
      break;
    case 3:
      e = launch_pdl(frame_cka_gate_kernel<3>, dim3(n_frames), dim3(kCkaThreads), 0, s, vbuf, abuf, n_frames, dim,
                     tau, beta, done, c_out, dbuf, s_out, dnorm_out, cbar_out);
      break;
    case 5:
      e = launch_pdl(frame_cka_gate_kernel<5>, dim3(n_frames), dim3(kCkaThreads), 0, s, vbuf, abuf, n_frames, dim,
                     tau, beta, done, c_out, dbuf, s_out, dnorm_out, cbar_out);
      break;
    default:
      e = launch_pdl(frame_cka_gate_kernel<7>, dim3(n_frames), dim3(kCkaThreads), 0, s, vbuf, abuf, n_frames, dim,
                     tau, beta, done, c_out, dbuf, s_out, dnorm_out, cbar_out);
      break;
  }
  count_launches(1);
  if (check_cuda(e) != APACK_OK) return APACK_ECUDA;
  return APACK_OK;
}

}  // extern "C"
