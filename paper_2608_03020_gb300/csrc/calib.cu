// One-shot reduced-rank fit of every block's feedback map from probe-backward pairs (Eq. 5;
// Theorem "Feedback ridge solution" and Lemma "Rank-truncation error", S5).  Untimed: it
// runs once, before Stage II.
//
// Token-major probe pairs: E_probe (Np x m) and G_probe_l (Np x d).
//   k_calib_xty    K = E^T E (m x m) and R_l = E^T G_l (m x d): fp32 products summed over
//                  32-token chunks, chunks accumulated in fp64.
//   k_calib_solve  per block l: Cholesky of K + beta I (fp64), F_l^T = (K + beta I)^-1 R_l by
//                  two triangular substitutions per column (no inverse), then the m x m matrix
//                  M = F^T F^T^T, its eigen-decomposition by cyclic Jacobi rotations (fp64),
//                  which gives the left singular vectors U and sigma = sqrt(eig) of F^T, and
//                  P_l = U_r S_r, Q_l = S_r^-1 U_r^T F^T = V_r^T.  Signs: the largest-magnitude
//                  entry of each Q row is made positive.  Singular values below 1e-12 sigma_1
//                  are treated as zero (zero Q row, zero P column).
#include <cuda_runtime.h>

#include "jacobi.cuh"
#include "loca_internal.h"

namespace loca {
namespace {

constexpr int XT_COLS = 64;
constexpr int XT_TOK = 32;

// out[b][s][j] = sum_n E[n][s] Y_b[n][j]   (s < m, j < w); Y_b = Y + b * Np * w
template <int KM>
__global__ void __launch_bounds__(256) k_calib_xty(const float* __restrict__ E, const float* __restrict__ Y,
                                                  int64_t Np, int m, int64_t w, double* __restrict__ out) {
  constexpr int SPT = KM / 4;  // s values per thread
  __shared__ float Es[XT_TOK][KM];
  __shared__ float Ys[XT_TOK][XT_COLS];
  const int b = blockIdx.y;
  const int jj = threadIdx.x % XT_COLS, grp = threadIdx.x / XT_COLS;
  const int64_t j = int64_t(blockIdx.x) * XT_COLS + jj;
  const float* Yb = Y + int64_t(b) * Np * w;
  double acc[SPT];
#pragma unroll
  for (int i = 0; i < SPT; ++i) acc[i] = 0.0;
  for (int64_t n0 = 0; n0 < Np; n0 += XT_TOK) {
    __syncthreads();
    for (int e = threadIdx.x; e < XT_TOK * KM; e += 256) {
      const int nn = e / KM, s = e % KM;
      Es[nn][s] = (n0 + nn < Np && s < m) ? E[(n0 + nn) * m + s] : 0.f;
    }
    for (int e = threadIdx.x; e < XT_TOK * XT_COLS; e += 256) {
      const int nn = e / XT_COLS, c = e % XT_COLS;
      const int64_t jc = int64_t(blockIdx.x) * XT_COLS + c;
      Ys[nn][c] = (n0 + nn < Np && jc < w && LOCA_CHECK((n0 + nn) * w + jc, Np * w)) ? Yb[(n0 + nn) * w + jc] : 0.f;
    }
    __syncthreads();
    float part[SPT];
#pragma unroll
    for (int i = 0; i < SPT; ++i) part[i] = 0.f;
#pragma unroll 4
    for (int nn = 0; nn < XT_TOK; ++nn) {
      const float yv = Ys[nn][jj];
#pragma unroll
      for (int i = 0; i < SPT; ++i) part[i] = fmaf(Es[nn][grp + 4 * i], yv, part[i]);
    }
#pragma unroll
    for (int i = 0; i < SPT; ++i) acc[i] += double(part[i]);
  }
  if (j >= w) return;
#pragma unroll
  for (int i = 0; i < SPT; ++i) {
    const int s = grp + 4 * i;
    if (s < m && LOCA_CHECK((int64_t(b) * m + s) * w + j, int64_t(gridDim.y) * m * w)) out[(int64_t(b) * m + s) * w + j] = acc[i];
  }
}

template <int KM>
struct CalibSmem {
  double Kc[KM][KM];  // K + beta I, then its Cholesky factor (lower)
  double A[KM][KM];   // F^T F^T^T, rotated towards diagonal
  double V[KM][KM];   // accumulated rotations (eigenvectors in columns)
  double red[256];
  int order[KM];
  int arg[256];
};

template <int KM>
__global__ void __launch_bounds__(256) k_calib_solve(const double* __restrict__ K, double* __restrict__ R,
                                                    int m, int64_t d, float beta, int r,
                                                    float* __restrict__ P, float* __restrict__ Q,
                                                    float* __restrict__ sigma, int32_t* status) {
  extern __shared__ __align__(16) unsigned char smem_raw[];
  CalibSmem<KM>& sm = *reinterpret_cast<CalibSmem<KM>*>(smem_raw);
  __shared__ int s_bad;
  const int l = blockIdx.x;
  const int t = threadIdx.x;
  double* F = R + int64_t(l) * m * d;  // R_l, overwritten with F_hat^T (m x d)

  for (int e = t; e < KM * KM; e += 256) {
    const int a = e / KM, b = e % KM;
    double v;
    if (a < m && b < m) {
      v = K[a * m + b];
      if (a == b) v += double(beta);
    } else {
      v = (a == b) ? 1.0 : 0.0;
    }
    sm.Kc[a][b] = v;
  }
  __syncthreads();
  // Cholesky of K + beta I (positive definite for beta > 0 in exact arithmetic; a pivot that is
  // not positive means beta is below the rounding level of E^T E: reported, outputs zeroed)
  if (t == 0) s_bad = 0;
  __syncthreads();
  if (t < 32) {
    for (int c = 0; c < KM; ++c) {
      double diag = sm.Kc[c][c];
      for (int u = 0; u < c; ++u) diag -= sm.Kc[c][u] * sm.Kc[c][u];
      if (!(diag > 0.0)) {
        if (t == 0) s_bad = 1;
        break;
      }
      const double lcc = sqrt(diag);
      __syncwarp();
      for (int rr = c + 1 + t; rr < KM; rr += 32) {
        double v = sm.Kc[rr][c];
        for (int u = 0; u < c; ++u) v -= sm.Kc[rr][u] * sm.Kc[c][u];
        sm.Kc[rr][c] = v / lcc;
      }
      __syncwarp();
      if (t == 0) sm.Kc[c][c] = lcc;
      __syncwarp();
    }
  }
  __syncthreads();
  if (s_bad) {
    if (t == 0) atomicExch(status, int32_t(LOCA_ERR_NUMERIC));
    if (!LOCA_CHECK_SPAN(int64_t(l) * r * d, int64_t(r) * d, int64_t(gridDim.x) * r * d)) return;
    for (int64_t e = t; e < int64_t(r) * d; e += 256) Q[int64_t(l) * r * d + e] = 0.f;
    for (int e = t; e < m * r; e += 256) P[int64_t(l) * m * r + e] = 0.f;
    if (sigma != nullptr)
      for (int e = t; e < r; e += 256) sigma[int64_t(l) * r + e] = 0.f;
    return;
  }
  // F^T[:, j] = (K + beta I)^-1 R[:, j]
  for (int64_t j = t; j < d; j += 256) {
    double x[KM];
#pragma unroll
    for (int s = 0; s < KM; ++s) x[s] = (s < m) ? F[int64_t(s) * d + j] : 0.0;
#pragma unroll
    for (int s = 0; s < KM; ++s) {
      double a = x[s];
#pragma unroll
      for (int u = 0; u < s; ++u) a -= sm.Kc[s][u] * x[u];
      x[s] = a / sm.Kc[s][s];
    }
#pragma unroll
    for (int s = KM - 1; s >= 0; --s) {
      double a = x[s];
#pragma unroll
      for (int u = s + 1; u < KM; ++u) a -= sm.Kc[u][s] * x[u];
      x[s] = a / sm.Kc[s][s];
    }
#pragma unroll
    for (int s = 0; s < KM; ++s)
      if (s < m) F[int64_t(s) * d + j] = x[s];
  }
  __syncthreads();
  // A = F^T (F^T)^T  (m x m), V = I
  for (int e = t; e < KM * KM; e += 256) {
    const int a = e / KM, b = e % KM;
    double v = 0.0;
    if (a < m && b < m && a <= b) {
      const double* fa = F + int64_t(a) * d;
      const double* fb = F + int64_t(b) * d;
      for (int64_t j = 0; j < d; ++j) v += fa[j] * fb[j];
    }
    sm.A[a][b] = v;
    sm.V[a][b] = (a == b) ? 1.0 : 0.0;
  }
  __syncthreads();
  for (int e = t; e < KM * KM; e += 256) {
    const int a = e / KM, b = e % KM;
    if (a > b) sm.A[a][b] = sm.A[b][a];
  }
  __syncthreads();
  // eigen-decomposition of F^T F^T^T by Jacobi rotations (whole block)
  jacobi_eig_block<KM>(sm.A, sm.V, sm.order, m);
  __syncthreads();
  const double lam1 = sm.A[sm.order[0]][sm.order[0]];
  const double s1 = lam1 > 0.0 ? sqrt(lam1) : 0.0;
  for (int i = 0; i < r; ++i) {
    const int col = sm.order[i];
    const double lam = (i < m) ? sm.A[col][col] : 0.0;
    double sg = lam > 0.0 ? sqrt(lam) : 0.0;
    if (!(sg > 1e-12 * s1)) sg = 0.0;
    float* qrow = Q + (int64_t(l) * r + i) * d;
    if (!LOCA_CHECK_SPAN((int64_t(l) * r + i) * d, d, int64_t(gridDim.x) * r * d)) break;
    // Q row = U_i^T F^T / sigma_i ; track the entry of largest magnitude (lowest index on ties)
    double best = -1.0;
    int64_t bj = 0;
    for (int64_t j = t; j < d; j += 256) {
      double v = 0.0;
      if (sg > 0.0) {
        for (int a = 0; a < m; ++a) v += sm.V[a][col] * F[int64_t(a) * d + j];
        v /= sg;
      }
      qrow[j] = float(v);
      if (fabs(v) > best) {
        best = fabs(v);
        bj = j;
      }
    }
    sm.red[t] = best;
    sm.arg[t] = int(bj);
    __syncthreads();
    for (int wdt = 128; wdt > 0; wdt >>= 1) {
      if (t < wdt) {
        const double o = sm.red[t + wdt];
        const int oa = sm.arg[t + wdt];
        if (o > sm.red[t] || (o == sm.red[t] && oa < sm.arg[t])) {
          sm.red[t] = o;
          sm.arg[t] = oa;
        }
      }
      __syncthreads();
    }
    const int64_t jmax = sm.arg[0];
    __syncthreads();
    const float sign = (qrow[jmax] < 0.f) ? -1.f : 1.f;
    __syncthreads();
    if (sign < 0.f)
      for (int64_t j = t; j < d; j += 256) qrow[j] = -qrow[j];
    for (int a = t; a < m; a += 256)
      if (LOCA_CHECK((int64_t(l) * m + a) * r + i, int64_t(gridDim.x) * m * r)) P[(int64_t(l) * m + a) * r + i] = float(sign * sm.V[a][col] * sg);
    if (sigma != nullptr && t == 0) sigma[int64_t(l) * r + i] = float(sg);
    __syncthreads();
  }
}

template <int KM>
cudaError_t calib_t(const float* E, const float* G, int64_t Np, int m, int64_t d, int L, float beta,
                    int r, float* P, float* Q, float* sigma, double* Kw, double* Rw, int32_t* status,
                    cudaStream_t s) {
  k_calib_xty<KM><<<dim3(unsigned((m + XT_COLS - 1) / XT_COLS), 1), 256, 0, s>>>(E, E, Np, m, m, Kw);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_calib_xty<KM><<<dim3(unsigned((d + XT_COLS - 1) / XT_COLS), unsigned(L)), 256, 0, s>>>(E, G, Np, m, d, Rw);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t shm = sizeof(CalibSmem<KM>);
  e = cudaFuncSetAttribute(k_calib_solve<KM>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
  if (e != cudaSuccess) return e;
  k_calib_solve<KM><<<L, 256, shm, s>>>(Kw, Rw, m, d, beta, r, P, Q, sigma, status);
  return cudaGetLastError();
}

}  // namespace

size_t calib_workspace_bytes(int64_t Np, int m, int64_t d, int L, int r) {
  (void)Np;
  (void)r;
  return align256(sizeof(double) * size_t(m) * size_t(m)) +
         align256(sizeof(double) * size_t(L) * size_t(m) * size_t(d));
}

cudaError_t launch_calib_fit(const float* E_probe, const float* G_probe, int64_t Np, int m, int64_t d,
                             int L, float beta, int r, float* P, float* Q, float* sigma, void* workspace,
                             int32_t* status, cudaStream_t s) {
  double* Kw = static_cast<double*>(workspace);
  double* Rw = reinterpret_cast<double*>(static_cast<char*>(workspace) +
                                         align256(sizeof(double) * size_t(m) * size_t(m)));
  if (m <= 8) return calib_t<8>(E_probe, G_probe, Np, m, d, L, beta, r, P, Q, sigma, Kw, Rw, status, s);
  if (m <= 16) return calib_t<16>(E_probe, G_probe, Np, m, d, L, beta, r, P, Q, sigma, Kw, Rw, status, s);
  if (m <= 32) return calib_t<32>(E_probe, G_probe, Np, m, d, L, beta, r, P, Q, sigma, Kw, Rw, status, s);
  return calib_t<64>(E_probe, G_probe, Np, m, d, L, beta, r, P, Q, sigma, Kw, Rw, status, s);
}

}  // namespace loca
