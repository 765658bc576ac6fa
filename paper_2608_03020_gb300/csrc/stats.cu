// Per-batch sum of squares, the scale-normalised step, and the exact-input (fp32) Gram /
// cross-product path.
//
// k_sumsq:      xsq_b[l] = ||X_l||_F^2 for this mini-batch (RMS of S8; trace of the batch Gram).
//               Grid (G, L): each thread block reduces a contiguous share of X_l with 16-byte
//               loads into one fp64 partial; k_step sums the G partials in a fixed order.
// k_step:       alpha_l = -eta sqrt(xsq_b / tsq) (= -eta_bar of Eq. 10, 0 when tsq == 0) and
//               xsq_total[l] (+)= xsq_b.
// k_step_from_gram: the same alpha_l and xsq_total[l] = xsq_b for a pass with one mini-batch,
//               with xsq_b = tr(Gram_l) = ||X_l||_F^2 read off the diagonal of that batch's Gram
//               (fp64 sum in a fixed order), so no separate read of X is needed.
// k_gram_cross_f32: Gram_l (+)= X^T X (upper tiles, mirrored) and Cross_l (+)= alpha T^T X for
//               fp32 inputs with fp64 accumulation: the exact-input path used for tight parity
//               on small shapes; the bf16 path runs on the tensor cores (gram_tc.cu).
#include <cuda_bf16.h>

#include "loca_internal.h"

namespace loca {
namespace {

constexpr int kMaxPartials = 1024;

template <bool kBF16>
__global__ void __launch_bounds__(256) k_sumsq(const void* __restrict__ Xv, int64_t N, int64_t d,
                                               int vec_ok, double* __restrict__ partials) {
  const int l = blockIdx.y;
  const int64_t n_el = N * d;
  const int64_t per = (n_el + gridDim.x - 1) / gridDim.x;
  int64_t beg = per * blockIdx.x;
  int64_t end = beg + per < n_el ? beg + per : n_el;
  double acc = 0.0;
  float part = 0.f;
  int cnt = 0;
  if (kBF16) {
    const __nv_bfloat16* X = static_cast<const __nv_bfloat16*>(Xv) + int64_t(l) * n_el;
    if (vec_ok) {
      // 8-element aligned interior
      int64_t vb = (beg + 7) / 8, ve = end / 8;
      for (int64_t e = beg + threadIdx.x; e < vb * 8 && e < end; e += blockDim.x) {
        if (!LOCA_CHECK(e, n_el)) break;
        const float v = __bfloat162float(X[e]);
        part = fmaf(v, v, part);
      }
      for (int64_t vi = vb + threadIdx.x; vi < ve; vi += blockDim.x) {
        if (!LOCA_CHECK_SPAN(vi * 8, 8, n_el)) break;
        const uint4 q = __ldg(reinterpret_cast<const uint4*>(X) + vi);
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          const float a = __uint_as_float(w[i] << 16), b = __uint_as_float(w[i] & 0xffff0000u);
          part = fmaf(a, a, part);
          part = fmaf(b, b, part);
        }
        if (++cnt == 4) { acc += part; part = 0.f; cnt = 0; }
      }
      for (int64_t e = (ve * 8 > vb * 8 ? ve * 8 : vb * 8) + threadIdx.x; e < end; e += blockDim.x) {
        if (!LOCA_CHECK(e, n_el)) break;
        const float v = __bfloat162float(X[e]);
        part = fmaf(v, v, part);
      }
    } else {
      for (int64_t e = beg + threadIdx.x; e < end; e += blockDim.x) {
        if (!LOCA_CHECK(e, n_el)) break;
        const float v = __bfloat162float(X[e]);
        part = fmaf(v, v, part);
        if (++cnt == 32) { acc += part; part = 0.f; cnt = 0; }
      }
    }
  } else {
    const float* X = static_cast<const float*>(Xv) + int64_t(l) * n_el;
    for (int64_t e = beg + threadIdx.x; e < end; e += blockDim.x) {
      if (!LOCA_CHECK(e, n_el)) break;
      const double v = X[e];
      acc = fma(v, v, acc);
    }
  }
  acc += part;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  __shared__ double red[8];
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double a = 0.0;
    for (int i = 0; i < int(blockDim.x >> 5); ++i) a += red[i];
    if (LOCA_CHECK(blockIdx.x, kMaxPartials)) partials[int64_t(l) * kMaxPartials + blockIdx.x] = a;
  }
}

__global__ void k_step(const double* __restrict__ partials, int G, int L, const double* __restrict__ tsq,
                       float eta, int zero_first, double* __restrict__ xsq_total,
                       float* __restrict__ alpha) {
  const int l = blockIdx.x * blockDim.x + threadIdx.x;
  if (l >= L || !LOCA_CHECK(G, kMaxPartials + 1)) return;
  double xb = 0.0;
  for (int g = 0; g < G; ++g) xb += partials[int64_t(l) * kMaxPartials + g];
  const double ts = tsq[l];
  alpha[l] = ts > 0.0 ? float(-double(eta) * sqrt(xb / ts)) : 0.f;
  xsq_total[l] = (zero_first ? 0.0 : xsq_total[l]) + xb;
}

__global__ void __launch_bounds__(256) k_step_from_gram(const float* __restrict__ gram, int64_t d,
                                                        const double* __restrict__ tsq, float eta,
                                                        double* __restrict__ xsq_total,
                                                        float* __restrict__ alpha) {
  __shared__ double red[8];
  const int l = blockIdx.x;
  const float* Gl = gram + int64_t(l) * d * d;
  double acc = 0.0;
  for (int64_t j = threadIdx.x; j < d; j += 256)
    if (LOCA_CHECK(j * (d + 1), d * d)) acc += double(Gl[j * (d + 1)]);
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double xb = 0.0;
    for (int w = 0; w < 8; ++w) xb += red[w];
    const double ts = tsq[l];
    alpha[l] = ts > 0.0 ? float(-double(eta) * sqrt(xb / ts)) : 0.f;
    xsq_total[l] = xb;
  }
}

// 64 x 64 output tile per thread block, 4 x 4 per thread, fp64 accumulators.
constexpr int FT = 64;
constexpr int FK = 16;

__global__ void __launch_bounds__(256) k_gram_cross_f32(const float* __restrict__ X,
                                                        const float* __restrict__ T, int64_t N,
                                                        int64_t d, const float* __restrict__ alpha,
                                                        int zero_first, float* __restrict__ gram,
                                                        float* __restrict__ cross) {
  const int l = blockIdx.z >> 1;
  const bool is_gram = (blockIdx.z & 1) == 0;
  const int mt = blockIdx.y, nt = blockIdx.x;
  if (is_gram && nt < mt) return;  // tile strictly below the diagonal: written by the mirror
  __shared__ float As[FK][FT];
  __shared__ float Bs[FK][FT];
  const float* Xl = X + int64_t(l) * N * d;
  const float* Rl = (is_gram ? X : T) + int64_t(l) * N * d;
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int64_t i0 = int64_t(mt) * FT, j0 = int64_t(nt) * FT;
  double acc[4][4] = {};
  for (int64_t n0 = 0; n0 < N; n0 += FK) {
    for (int e = threadIdx.x; e < FK * FT; e += 256) {
      const int kk = e / FT, c = e % FT;
      const int64_t n = n0 + kk;
      As[kk][c] = (n < N && i0 + c < d && LOCA_CHECK(n * d + i0 + c, N * d)) ? Rl[n * d + i0 + c] : 0.f;
      Bs[kk][c] = (n < N && j0 + c < d && LOCA_CHECK(n * d + j0 + c, N * d)) ? Xl[n * d + j0 + c] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < FK; ++kk) {
      double a[4], b[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) a[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) b[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fma(a[i], b[j], acc[i][j]);
    }
    __syncthreads();
  }
  const double al = is_gram ? 1.0 : double(alpha[l]);
  float* out = (is_gram ? gram : cross) + int64_t(l) * d * d;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int64_t r = i0 + ty * 4 + i;
    if (r >= d) continue;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int64_t c = j0 + tx * 4 + j;
      if (c >= d) continue;
      if (is_gram && r > c) continue;
      if (!LOCA_CHECK(r * d + c, d * d) || !LOCA_CHECK(c * d + r, d * d)) continue;
      const double v = al * acc[i][j];
      float* p = out + r * d + c;
      *p = zero_first ? float(v) : float(double(*p) + v);
      if (is_gram && r < c) {
        float* q = out + c * d + r;
        *q = zero_first ? float(v) : float(double(*q) + v);
      }
    }
  }
}

}  // namespace

int sumsq_num_partials() { return kMaxPartials; }

cudaError_t launch_sumsq_and_step(const void* X, int dtype, int L, int64_t N, int64_t d,
                                  const double* tsq, float eta, int zero_first, double* xsq_total,
                                  double* partials, float* alpha, cudaStream_t s) {
  int64_t G = (int64_t(sm_count()) * 8 + L - 1) / L;
  const int64_t n_el = N * d;
  const int64_t maxg = (n_el + 4095) / 4096;  // at least 4096 elements per thread block
  if (G > maxg) G = maxg;
  if (G < 1) G = 1;
  if (G > kMaxPartials) G = kMaxPartials;
  if (n_el > 0) {
    const dim3 grid = dim3(unsigned(G), unsigned(L));
    if (dtype == LOCA_BF16) {
      const int vec_ok = (reinterpret_cast<uintptr_t>(X) % 16 == 0) && (n_el % 8 == 0);
      k_sumsq<true><<<grid, 256, 0, s>>>(X, N, d, vec_ok, partials);
    } else {
      k_sumsq<false><<<grid, 256, 0, s>>>(X, N, d, 0, partials);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  } else {
    G = 0;
  }
  k_step<<<(L + 127) / 128, 128, 0, s>>>(partials, int(G), L, tsq, eta, zero_first, xsq_total, alpha);
  return cudaGetLastError();
}

cudaError_t launch_gram_cross_f32(const float* X, const float* T, int L, int64_t N, int64_t d,
                                  const float* alpha, int zero_first, float* gram, float* cross,
                                  cudaStream_t s) {
  const unsigned nt = unsigned((d + FT - 1) / FT);
  const dim3 grid = dim3(nt, nt, unsigned(2 * L));
  k_gram_cross_f32<<<grid, 256, 0, s>>>(X, T, N, d, alpha, zero_first, gram, cross);
  return cudaGetLastError();
}

cudaError_t launch_step_from_gram(const float* gram, int L, int64_t d, const double* tsq, float eta,
                                  double* xsq_total, float* alpha, cudaStream_t s) {
  k_step_from_gram<<<L, 256, 0, s>>>(gram, d, tsq, eta, xsq_total, alpha);
  return cudaGetLastError();
}

}  // namespace loca
