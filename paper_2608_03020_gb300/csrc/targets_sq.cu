// ||T_l||_F^2 of the feedback targets T_l = (E P_l) Q_l (S3, S11) without forming T_l:
//   ||T_l||^2 = sum_n u_n^T (Q_l Q_l^T) u_n,  u_n = e_n P_l
//             = < P_l (Q_l Q_l^T) P_l^T , E^T E >   (Frobenius inner product of two C x C matrices).
// The step of Eq. 10 needs it when the statistics kernel generates T itself (fused targets).
//
// k_tsq_ete    partial E^T E over chunks of TSQ_CHUNK tokens (fp32 products summed in fp64), one
//              C x C slot per chunk.
// k_tsq_block  one CTA per block l: the chunks' slots summed in a fixed order, M_l = Q_l Q_l^T
//              (fp32 products over runs of 32 channels, runs summed in fp64), K = P_l M_l P_l^T and
//              <K, E^T E> in fp64.  Deterministic.
#include "loca_internal.h"

namespace loca {
namespace {

constexpr int TSQ_THREADS = 256;
constexpr int TSQ_CHUNK = 2048;  // tokens per E^T E partial
constexpr int kMaxC = 64;
constexpr int kMaxR = 32;

__global__ void __launch_bounds__(TSQ_THREADS) k_tsq_ete(const float* __restrict__ E, int64_t N, int C,
                                                          double* __restrict__ part) {
  const int64_t n0 = int64_t(blockIdx.x) * TSQ_CHUNK;
  const int64_t n1 = n0 + TSQ_CHUNK < N ? n0 + TSQ_CHUNK : N;
  double* out = part + int64_t(blockIdx.x) * C * C;
  for (int e = threadIdx.x; e < C * C; e += TSQ_THREADS) {
    const int a = e / C, b = e % C;
    double acc = 0.0;
    for (int64_t n = n0; n < n1; ++n)
      if (LOCA_CHECK(n * C + a, N * C) && LOCA_CHECK(n * C + b, N * C)) acc += double(E[n * C + a]) * double(E[n * C + b]);
    if (LOCA_CHECK(int64_t(blockIdx.x) * C * C + e, int64_t(gridDim.x) * C * C)) out[e] = acc;
  }
}

__global__ void __launch_bounds__(TSQ_THREADS) k_tsq_block(const double* __restrict__ part, int nchunks, int C,
                                                            const float* __restrict__ P, const float* __restrict__ Q,
                                                            int r, int64_t d, double* __restrict__ tsq) {
  __shared__ double ete[kMaxC * kMaxC];
  __shared__ double M[kMaxR * kMaxR];
  __shared__ double PM[kMaxC * kMaxR];
  __shared__ double red[TSQ_THREADS];
  const int l = blockIdx.x;
  for (int e = threadIdx.x; e < C * C; e += TSQ_THREADS) {
    double acc = 0.0;
    for (int c = 0; c < nchunks; ++c) acc += part[int64_t(c) * C * C + e];  // e < C * C
    ete[e] = acc;
  }
  // M = Q_l Q_l^T: one warp per entry (s, t), lanes over channels, fp32 runs of 32 products
  const float* Ql = Q + int64_t(l) * r * d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int e = warp; e < r * r; e += TSQ_THREADS / 32) {
    const int si = e / r, ti = e % r;
    if (ti < si) continue;
    const float* qs = Ql + int64_t(si) * d;
    const float* qt = Ql + int64_t(ti) * d;
    double acc = 0.0;
    for (int64_t c0 = 0; c0 < d; c0 += 32 * 32) {
      float run = 0.f;
      for (int64_t c = c0 + lane; c < c0 + 32 * 32 && c < d; c += 32) run = fmaf(qs[c], qt[c], run);
      acc += double(run);
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) {
      M[si * r + ti] = acc;
      M[ti * r + si] = acc;
    }
  }
  __syncthreads();
  // PM = P_l M (C x r)
  const float* Pl = P + int64_t(l) * C * r;
  for (int e = threadIdx.x; e < C * r; e += TSQ_THREADS) {
    const int a = e / r, t = e % r;
    double acc = 0.0;
    for (int s = 0; s < r; ++s) acc += double(Pl[a * r + s]) * M[s * r + t];
    PM[e] = acc;
  }
  __syncthreads();
  // <P M P^T, E^T E> = sum_ab (sum_t PM[a, t] P[b, t]) ete[a, b]
  double acc = 0.0;
  for (int e = threadIdx.x; e < C * C; e += TSQ_THREADS) {
    const int a = e / C, b = e % C;
    double k = 0.0;
    for (int t = 0; t < r; ++t) k += PM[a * r + t] * double(Pl[b * r + t]);
    acc += k * ete[e];
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  for (int w = TSQ_THREADS / 2; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0 && LOCA_CHECK(l, gridDim.x)) tsq[l] = red[0];
}

}  // namespace

int tsq_max_C() { return kMaxC; }
int tsq_max_r() { return kMaxR; }

size_t tsq_workspace_bytes(int64_t N, int C) {
  const int64_t nchunks = (N + TSQ_CHUNK - 1) / TSQ_CHUNK;
  return align256(sizeof(double) * size_t(nchunks > 0 ? nchunks : 1) * size_t(C) * size_t(C));
}

cudaError_t launch_targets_sq(const float* E, int64_t N, int C, const float* P, const float* Q, int L, int r,
                              int64_t d, double* tsq, void* workspace, cudaStream_t s) {
  const int64_t nchunks = (N + TSQ_CHUNK - 1) / TSQ_CHUNK;
  double* part = static_cast<double*>(workspace);
  if (nchunks > 0) k_tsq_ete<<<unsigned(nchunks), TSQ_THREADS, 0, s>>>(E, N, C, part);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_tsq_block<<<unsigned(L), TSQ_THREADS, 0, s>>>(part, int(nchunks), C, P, Q, r, d, tsq);
  return cudaGetLastError();
}

}  // namespace loca
