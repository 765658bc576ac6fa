// Symmetric eigen-decomposition by Jacobi rotations (fp64, one thread block), shared by the
// calibration kernels: the thin SVD F^T = U S V^T of the feedback fit (Lemma "Rank-truncation
// error", S5) is read off the eigen-decomposition of a small Gram matrix (U, S^2).
#pragma once

#include <cuda_runtime.h>

namespace loca {

// A (m x m, symmetric, shared memory with row stride KM) is rotated towards diagonal form and
// V (initialised by the caller, usually to I) accumulates the rotations, so that on return the
// columns of V are eigenvectors and diag(A) the eigenvalues.
//
// Parallel ordering: a sweep is m - 1 rounds (m rounded up to even, the extra index a dummy) of
// a round-robin tournament, so that every pair (p, q) meets once per sweep and the m / 2 pairs
// of a round are disjoint; their rotations are applied at once, to rows (A <- J^T A), then to
// columns (A <- A J, V <- V J).  The rotation of pair (p, q) has tan(phi) = t, the root of
// smaller magnitude of t^2 + 2 theta t - 1 = 0 with theta = (A_qq - A_pp) / (2 A_pq), which
// zeroes (J^T A J)_pq.  Sweeps stop when the off-diagonal mass falls below 1e-30 of the total,
// after at most 40 sweeps.  Then order[] = eigenvalue indices in descending order (stable:
// lower index first on ties; entries m..KM-1 stay in place).  Called by every thread of the
// block (it synchronises the block).
template <int KM>
__device__ void jacobi_eig_block(double (*A)[KM], double (*V)[KM], int* order, int m) {
  __shared__ double s_c[KM / 2], s_s[KM / 2];
  __shared__ int s_p[KM / 2], s_q[KM / 2];
  __shared__ int s_go;
  const int tid = threadIdx.x, nt = blockDim.x;
  const int mm = (m + 1) & ~1;
  const int np = mm / 2;
  for (int sweep = 0; sweep < 40; ++sweep) {
    __syncthreads();
    if (tid == 0) {
      double off = 0.0, total = 0.0;
      for (int a = 0; a < m; ++a)
        for (int b = 0; b < m; ++b) {
          const double v = A[a][b] * A[a][b];
          total += v;
          if (a != b) off += v;
        }
      s_go = (off > 1e-30 * total) ? 1 : 0;
    }
    __syncthreads();
    if (!s_go) break;
    for (int k = 0; k < mm - 1; ++k) {
      if (tid < np) {
        int p, q;
        if (tid == 0) {
          p = k % (mm - 1);
          q = mm - 1;
        } else {
          p = (k + tid) % (mm - 1);
          q = (k - tid + mm - 1) % (mm - 1);
        }
        if (p > q) {
          const int tmp = p;
          p = q;
          q = tmp;
        }
        double c = 1.0, sn = 0.0;
        if (q < m) {
          const double apq = A[p][q];
          if (fabs(apq) > 1e-300) {
            const double theta = (A[q][q] - A[p][p]) / (2.0 * apq);
            const double t = (theta >= 0 ? 1.0 : -1.0) / (fabs(theta) + sqrt(theta * theta + 1.0));
            c = 1.0 / sqrt(t * t + 1.0);
            sn = t * c;
          }
        }
        s_p[tid] = p;
        s_q[tid] = q;
        s_c[tid] = c;
        s_s[tid] = sn;
      }
      __syncthreads();
      for (int e = tid; e < np * m; e += nt) {
        const int i = e / m, col = e % m;
        const int p = s_p[i], q = s_q[i];
        if (q >= m) continue;
        const double c = s_c[i], sn = s_s[i];
        const double apk = A[p][col], aqk = A[q][col];
        A[p][col] = c * apk - sn * aqk;
        A[q][col] = sn * apk + c * aqk;
      }
      __syncthreads();
      for (int e = tid; e < np * m; e += nt) {
        const int i = e / m, row = e % m;
        const int p = s_p[i], q = s_q[i];
        if (q >= m) continue;
        const double c = s_c[i], sn = s_s[i];
        const double akp = A[row][p], akq = A[row][q];
        A[row][p] = c * akp - sn * akq;
        A[row][q] = sn * akp + c * akq;
        const double vkp = V[row][p], vkq = V[row][q];
        V[row][p] = c * vkp - sn * vkq;
        V[row][q] = sn * vkp + c * vkq;
      }
      __syncthreads();
      if (tid < np && s_q[tid] < m) {
        A[s_p[tid]][s_q[tid]] = 0.0;
        A[s_q[tid]][s_p[tid]] = 0.0;
      }
      __syncthreads();
    }
  }
  if (tid == 0) {
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
  __syncthreads();
}

}  // namespace loca
