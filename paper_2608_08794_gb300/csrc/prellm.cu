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
//  gate kernel:  one CTA: c-bar, min/max of d, the min-max normalised distance and the
//                gated score s_f of Eq. gate (blend when c-bar < tau).
// All reductions run in a fixed order: results are deterministic.
#include <cmath>

#include "internal.cuh"

namespace apack {

namespace {

constexpr int kPoolThreads = 256;      // 8 features per thread: 2048 features per CTA
constexpr int kCkaThreads = 256;
constexpr int kMaxWindow = 7;
constexpr int kGram = kMaxWindow * (kMaxWindow + 1) / 2;   // upper triangle of a w x w Gram
constexpr int kGateThreads = 1024;

__device__ __forceinline__ void add_bf16x8(const uint4 &v, float (&acc)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    acc[2 * i] += __uint_as_float(w[i] << 16);
    acc[2 * i + 1] += __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__global__ void __launch_bounds__(kPoolThreads)
    frame_pool_kernel(const uint4 *__restrict__ visual, const uint4 *__restrict__ audio, int n_frames, int tpf,
                      int n_audio, int64_t dim, float *__restrict__ v_out, float *__restrict__ a_out) {
  const int f = blockIdx.x;
  const int64_t fi = (static_cast<int64_t>(blockIdx.y) * kPoolThreads + threadIdx.x) * 8;
  if (fi >= dim) return;
  const int64_t vec_per_row = dim / 8;
  const int64_t col = fi / 8;
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  const int64_t r0 = static_cast<int64_t>(f) * tpf;
#pragma unroll 4
  for (int t = 0; t < tpf; ++t) add_bf16x8(__ldg(visual + (r0 + t) * vec_per_row + col), acc);
  const float inv_v = 1.f / static_cast<float>(tpf);
#pragma unroll
  for (int i = 0; i < 8; ++i) v_out[static_cast<int64_t>(f) * dim + fi + i] = acc[i] * inv_v;
  // audio tokens j with floor(j F / N_a) == f: j in [ceil(f N_a / F), ceil((f+1) N_a / F))
  const int64_t j0 = (static_cast<int64_t>(f) * n_audio + n_frames - 1) / n_frames;
  const int64_t j1 = (static_cast<int64_t>(f + 1) * n_audio + n_frames - 1) / n_frames;
#pragma unroll
  for (int i = 0; i < 8; ++i) acc[i] = 0.f;
#pragma unroll 4
  for (int64_t j = j0; j < j1; ++j) add_bf16x8(__ldg(audio + j * vec_per_row + col), acc);
  const float inv_a = 1.f / static_cast<float>(j1 - j0);
#pragma unroll
  for (int i = 0; i < 8; ++i) a_out[static_cast<int64_t>(f) * dim + fi + i] = acc[i] * inv_a;
}

__global__ void __launch_bounds__(kCkaThreads)
    frame_cka_kernel(const float *__restrict__ v, const float *__restrict__ a, int n_frames, int64_t dim, int window,
                     float *__restrict__ c_out, float *__restrict__ d_out) {
  __shared__ float red[kCkaThreads / 32][2 * kGram + 1];
  const int f = blockIdx.x;
  const int half = window / 2;
  const int lo = max(0, f - half), hi = min(n_frames, f + half + 1);
  const int w = hi - lo;
  const int center = f - lo;
  float ga[kGram], gv[kGram], dist = 0.f;
#pragma unroll
  for (int i = 0; i < kGram; ++i) ga[i] = gv[i] = 0.f;
  for (int64_t x = threadIdx.x; x < dim; x += kCkaThreads) {
    float av[kMaxWindow], vv[kMaxWindow], am = 0.f, vm = 0.f;
#pragma unroll
    for (int r = 0; r < kMaxWindow; ++r) {
      av[r] = r < w ? a[static_cast<int64_t>(lo + r) * dim + x] : 0.f;
      vv[r] = r < w ? v[static_cast<int64_t>(lo + r) * dim + x] : 0.f;
      am += av[r];
      vm += vv[r];
    }
    {
      const float dd = vv[center] - av[center];
      dist = fmaf(dd, dd, dist);
    }
    am /= static_cast<float>(w);
    vm /= static_cast<float>(w);
#pragma unroll
    for (int r = 0; r < kMaxWindow; ++r) {
      av[r] = r < w ? av[r] - am : 0.f;
      vv[r] = r < w ? vv[r] - vm : 0.f;
    }
    int k = 0;
#pragma unroll
    for (int i = 0; i < kMaxWindow; ++i)
#pragma unroll
      for (int j = i; j < kMaxWindow; ++j, ++k) {
        ga[k] = fmaf(av[i], av[j], ga[k]);
        gv[k] = fmaf(vv[i], vv[j], gv[k]);
      }
  }
  // block reduction of the 2 * kGram + 1 sums (warp tree, then warps in order)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int i = 0; i < kGram; ++i) {
    for (int o = 16; o > 0; o >>= 1) {
      ga[i] += __shfl_xor_sync(0xffffffffu, ga[i], o);
      gv[i] += __shfl_xor_sync(0xffffffffu, gv[i], o);
    }
  }
  for (int o = 16; o > 0; o >>= 1) dist += __shfl_xor_sync(0xffffffffu, dist, o);
  if (lane == 0) {
#pragma unroll
    for (int i = 0; i < kGram; ++i) {
      red[warp][i] = ga[i];
      red[warp][kGram + i] = gv[i];
    }
    red[warp][2 * kGram] = dist;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double sa[kGram], sv[kGram], sd = 0.0;
    for (int i = 0; i < kGram; ++i) {
      sa[i] = sv[i] = 0.0;
      for (int wp = 0; wp < kCkaThreads / 32; ++wp) {
        sa[i] += red[wp][i];
        sv[i] += red[wp][kGram + i];
      }
    }
    for (int wp = 0; wp < kCkaThreads / 32; ++wp) sd += red[wp][2 * kGram];
    // <K_A, K_V>_F, ||K_A||_F^2, ||K_V||_F^2 from the upper triangles
    double dot = 0.0, na = 0.0, nv = 0.0;
    int k = 0;
    for (int i = 0; i < kMaxWindow; ++i)
      for (int j = i; j < kMaxWindow; ++j, ++k) {
        if (i >= w || j >= w) continue;
        const double m = (i == j) ? 1.0 : 2.0;
        dot += m * sa[k] * sv[k];
        na += m * sa[k] * sa[k];
        nv += m * sv[k] * sv[k];
      }
    const double den = sqrt(na) * sqrt(nv);
    c_out[f] = den > 0.0 ? static_cast<float>(dot / den) : 0.f;
    d_out[f] = static_cast<float>(sqrt(sd));
  }
}

__global__ void __launch_bounds__(kGateThreads)
    frame_gate_kernel(const float *__restrict__ c, const float *__restrict__ d, int n_frames, float tau, float beta,
                      float *__restrict__ s_out, float *__restrict__ dn_out, float *__restrict__ cbar_out) {
  __shared__ double rsum[kGateThreads / 32];
  __shared__ float rmin[kGateThreads / 32], rmax[kGateThreads / 32];
  __shared__ double cbar_s;
  __shared__ float dmin_s, dmax_s;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  double cs = 0.0;
  float mn = INFINITY, mx = -INFINITY;
  for (int f = threadIdx.x; f < n_frames; f += kGateThreads) {
    cs += c[f];
    mn = fminf(mn, d[f]);
    mx = fmaxf(mx, d[f]);
  }
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
    float a = INFINITY, b = -INFINITY;
    for (int wp = 0; wp < kGateThreads / 32; ++wp) {
      t += rsum[wp];
      a = fminf(a, rmin[wp]);
      b = fmaxf(b, rmax[wp]);
    }
    cbar_s = t / n_frames;
    dmin_s = a;
    dmax_s = b;
    if (cbar_out) *cbar_out = static_cast<float>(cbar_s);
  }
  __syncthreads();
  const bool blend = cbar_s < static_cast<double>(tau);
  const float span = dmax_s - dmin_s;
  for (int f = threadIdx.x; f < n_frames; f += kGateThreads) {
    const float dn = span > 0.f ? (d[f] - dmin_s) / span : 0.f;
    if (dn_out) dn_out[f] = dn;
    s_out[f] = blend ? (1.f - beta) * c[f] + beta * (1.f - dn) : c[f];
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
  float *vbuf = reinterpret_cast<float *>(w + 256);
  float *abuf = reinterpret_cast<float *>(w + 256 + up(static_cast<size_t>(n_frames) * dim * sizeof(float)));
  float *dbuf = reinterpret_cast<float *>(w + 256 + 2 * up(static_cast<size_t>(n_frames) * dim * sizeof(float)));
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  dim3 pgrid(n_frames, static_cast<unsigned>((dim + kPoolThreads * 8 - 1) / (kPoolThreads * 8)));
  frame_pool_kernel<<<pgrid, kPoolThreads, 0, s>>>(static_cast<const uint4 *>(visual), static_cast<const uint4 *>(audio),
                                                  n_frames, tokens_per_frame, n_audio, dim, vbuf, abuf);
  count_launches(1);
  if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  frame_cka_kernel<<<n_frames, kCkaThreads, 0, s>>>(vbuf, abuf, n_frames, dim, window, c_out, dbuf);
  count_launches(1);
  if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  frame_gate_kernel<<<1, kGateThreads, 0, s>>>(c_out, dbuf, n_frames, tau, beta, s_out, dnorm_out, cbar_out);
  count_launches(1);
  if (check_cuda(cudaGetLastError()) != APACK_OK) return APACK_ECUDA;
  return APACK_OK;
}

}  // extern "C"
