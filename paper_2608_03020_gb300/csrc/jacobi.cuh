// Symmetric eigen-decomposition by cyclic Jacobi rotations (fp64, one warp), shared by the
// calibration kernels: the thin SVD F^T = U S V^T of the feedback fit (Lemma "Rank-truncation
// error", S5) is read off the eigen-decomposition of a small Gram matrix (U, S^2).
#pragma once

#include <cuda_runtime.h>

namespace loca {

// A (m x m, symmetric, shared memory with row stride KM) is rotated towards diagonal form and
// V (initialised by the caller, usually to I) accumulates the rotations, so that on return the
// columns of V are eigenvectors and diag(A) the eigenvalues.  Each rotation J in the (p, q)
// plane has tan(phi) = t with t^2 + 2 theta t - 1 = 0, theta = (A_qq - A_pp) / (2 A_pq), the
// root of smaller magnitude, which zeroes (J^T A J)_pq.  Sweeps stop when the off-diagonal mass
// falls below 1e-30 of the total, after at most 40 sweeps.  Lane 0 then writes order[] =
// eigenvalue indices in descending order (stable: lower index first on ties; entries m..KM-1
// stay in place).  Called by the 32 lanes of one warp.
template <int KM>
__device__ void jacobi_eig_warp(double (*A)[KM], double (*V)[KM], int* order, int m, int lane) {
  double total = 0.0;
  for (int a = 0; a < m; ++a)
    for (int b = 0; b < m; ++b) total += A[a][b] * A[a][b];
  for (int sweep = 0; sweep < 40; ++sweep) {
    double off = 0.0;
    for (int a = 0; a < m; ++a)
      for (int b = a + 1; b < m; ++b) off += A[a][b] * A[a][b];
    if (!(off > 1e-30 * total)) break;
    for (int p = 0; p < m - 1; ++p) {
      for (int q = p + 1; q < m; ++q) {
        const double apq = A[p][q];
        if (fabs(apq) <= 1e-300) continue;
        const double theta = (A[q][q] - A[p][p]) / (2.0 * apq);
        const double tt = (theta >= 0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
        const double c = 1.0 / sqrt(tt * tt + 1.0), s = tt * c;
        __syncwarp();
        for (int k = lane; k < m; k += 32) {
          if (k != p && k != q) {
            const double akp = A[k][p], akq = A[k][q];
            A[k][p] = c * akp - s * akq;
            A[k][q] = s * akp + c * akq;
          }
          const double vkp = V[k][p], vkq = V[k][q];
          V[k][p] = c * vkp - s * vkq;
          V[k][q] = s * vkp + c * vkq;
        }
        __syncwarp();
        for (int k = lane; k < m; k += 32) {
          if (k != p && k != q) {
            A[p][k] = A[k][p];
            A[q][k] = A[k][q];
          }
        }
        if (lane == 0) {
          A[p][p] -= tt * apq;
          A[q][q] += tt * apq;
          A[p][q] = 0.0;
          A[q][p] = 0.0;
        }
        __syncwarp();
      }
    }
  }
  if (lane == 0) {
    for (int i = 0; i < KM; ++i) order[i] = i;
    for (int i = 0; i < m; ++i) {
      int best = i;
      for (int k = i + 1; k < m; ++k)
        if (A[order[k]][order[k]] > A[order[best]][order[best]]) best = k;
      const int tmp = order[i];
      order[i] = order[best];
      order[best] = tmp;
    }
  }
  __syncwarp();
}

}  // namespace loca
