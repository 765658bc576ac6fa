// Small positive-definite solves shared by the ridge-solve kernels (S7: no explicit inverse).
//
// The k x k system matrix (k <= KM) lives in shared memory in fp64, padded to KM x KM with an
// identity block; warp 0 factors it (Cholesky, lower, column by column); every thread then
// solves its own right-hand side row by a forward and a back substitution in fp32 registers.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace loca {

// Factor Md = L L^T in place (lower triangle) with warp 0; then every thread of the block
// fills Lf (fp32 lower factor) and Linv (fp32 reciprocals of its diagonal).  Returns 0, or
// c + 1 when the leading minor of order c + 1 is not positive definite.  Must be called by
// every thread of the block (it synchronises the block).
template <int KM>
__device__ int chol_factor(double (*Md)[KM], float (*Lf)[KM], float* Linv, int* s_info) {
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    int inf = 0;
    for (int c = 0; c < KM; ++c) {
      double diag = Md[c][c];
      for (int t = 0; t < c; ++t) diag -= Md[c][t] * Md[c][t];
      if (!(diag > 0.0)) {
        inf = c + 1;
        break;
      }
      const double lcc = sqrt(diag);
      __syncwarp();
      for (int r = c + 1 + lane; r < KM; r += 32) {
        double v = Md[r][c];
        for (int t = 0; t < c; ++t) v -= Md[r][t] * Md[c][t];
        Md[r][c] = v / lcc;
      }
      __syncwarp();
      if (lane == 0) Md[c][c] = lcc;
      __syncwarp();
    }
    if (lane == 0) *s_info = inf;
  }
  __syncthreads();
  const int inf = *s_info;
  for (int e = threadIdx.x; e < KM * KM; e += blockDim.x) {
    const int a = e / KM, b = e % KM;
    Lf[a][b] = (b <= a && inf == 0) ? float(Md[a][b]) : 0.f;
  }
  for (int a = threadIdx.x; a < KM; a += blockDim.x) Linv[a] = inf == 0 ? float(1.0 / Md[a][a]) : 0.f;
  __syncthreads();
  return inf;
}

// c <- c (L L^T)^-1 for one row c (length KM) in registers.
template <int KM>
__device__ __forceinline__ void chol_solve_row(const float (*Lf)[KM], const float* Linv, float* c) {
#pragma unroll
  for (int s = 0; s < KM; ++s) {
    float a = c[s];
#pragma unroll
    for (int t = 0; t < s; ++t) a = fmaf(-Lf[s][t], c[t], a);
    c[s] = a * Linv[s];
  }
#pragma unroll
  for (int s = KM - 1; s >= 0; --s) {
    float a = c[s];
#pragma unroll
    for (int t = s + 1; t < KM; ++t) a = fmaf(-Lf[t][s], c[t], a);
    c[s] = a * Linv[s];
  }
}

}  // namespace loca
