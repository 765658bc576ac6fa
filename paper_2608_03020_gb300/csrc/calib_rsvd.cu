// Rank-r feedback fit for wide error spaces (Eq. 5; Theorem "Feedback ridge solution" and
// Lemma "Rank-truncation error", S5) when the error width m is too large to form and
// decompose F_hat_l^T = (E^T E + beta I_m)^-1 E^T G_l (m x d), e.g. the paper's e = W_u^T eps
// with m = d.  The top-r SVD comes from randomized subspace iteration (Halko, Martinsson and
// Tropp, SIAM Review 53 (2011), Algorithm 4.4, then Algorithm 5.1 on the projected matrix),
// which only applies F_hat^T and F_hat to blocks of ell vectors:
//
//   F^T X = K^-1 E^T (G_l X),   F Y = G_l^T E (K^-1 Y),   K = E^T E + beta I  (never inverted:
//   a Cholesky factor and two triangular solves per application).
//
// All L blocks share K, so every solve runs on the ell columns of all blocks at once.
//
//   k_cr_gemm     fp32 operands, products summed in fp32 over 32 terms, those sums in fp32 over
//                 16 and in fp64 beyond (the products with E and G_l; K itself, lower tiles only)
//   k_cr_pad      K + beta I, padded to a multiple of 64 with an identity block
//   k_cr_potrf / k_cr_trsm / k_cr_syrk   right-looking blocked Cholesky (64 x 64 tiles, fp64);
//                 the diagonal kernel also inverts its triangular tile, so the panel and the
//                 diagonal steps of the solves are tile products
//   k_cr_tsolve   blocked forward (L Y = W) and backward (L^T X = Y) substitution: fp64 for the
//                 last F^T (which makes the final basis Q_Y) and for the Rayleigh-Ritz product
//                 F Q_Y; fp32 (on an fp32 copy of the fp64 factor) inside the power iterations,
//                 which only steer the subspace: an error there moves the starting vectors of
//                 the next step, and the exact last F^T damps it by sigma_{ell+1} / sigma_r
//   k_cr_vtv / k_cr_qr_factor / k_cr_qr_apply
//                 orthonormal basis of each block's ell columns by Cholesky QR, applied twice
//                 (fp64): S = V^T V over row chunks on all SMs, S = R^T R, V <- V R^-1.  A column
//                 whose component outside the span of the earlier ones is below 1e-7 of its norm
//                 is dependent and set to zero
//   k_cr_btb / k_cr_ritz_eig / k_cr_ritz_out / k_cr_ritz_sign
//                 Rayleigh-Ritz: B^T = F Q_Y (d x ell), B B^T = U_B S^2 U_B^T by cyclic Jacobi,
//                 P_l = Q_Y U_B,r S_r, Q_l = S_r^-1 U_B,r^T B; the entry of largest magnitude of
//                 each Q_l row is made positive; singular values <= 1e-12 sigma_1 count as zero.
#include <cuda_runtime.h>

#include "jacobi.cuh"
#include "loca_internal.h"

namespace loca {
namespace {

constexpr int NB = 64;        // Cholesky / solve tile
constexpr int NBP = NB + 1;   // padded shared-memory row (fp64: conflict-free column reads)
constexpr int GM_BM = 64, GM_BN = 64, GM_BK = 32, GM_RUN = 16;
constexpr int RZ_CH = 256;    // rows per chunk of the Rayleigh-Ritz kernels
constexpr int kMaxEll = 64;
constexpr int64_t kMaxWidth = 16384;  // m and d (fp64 vectors of one column in shared memory)
constexpr size_t kTileSmem = sizeof(double) * 2 * NB * NBP;

__device__ __forceinline__ bool failed(const int32_t* flag) { return *reinterpret_cast<const volatile int32_t*>(flag) != 0; }

// C_b[i][j] = sum_t A_b(i, t) B_b(t, j);  A_b(i, t) = A[t lda + i] (AT) or A[i lda + t];
// B_b(t, j) = B[t ldb + j]; batch b = blockIdx.z with element strides sA, sB, sC.  Products are
// summed in fp32 over 32 terms, those sums in fp32 over 16 (512 terms), and those in fp64.  The
// next 32-term slab is loaded into registers while the current one is multiplied, then stored
// to the other shared-memory buffer (one barrier per slab).
template <bool AT, typename TC>
__global__ void __launch_bounds__(256) k_cr_gemm(const float* __restrict__ A, int64_t lda, int64_t sA,
                                                const float* __restrict__ B, int64_t ldb, int64_t sB,
                                                TC* __restrict__ C, int64_t ldc, int64_t sC, int64_t M, int64_t N,
                                                int64_t Kc, int lower_only) {
  __shared__ __align__(16) float As[2][GM_BK][GM_BM + 4];
  __shared__ __align__(16) float Bs[2][GM_BK][GM_BN + 4];
  constexpr int LPT = GM_BK * GM_BM / 256;
  const int64_t i0 = int64_t(blockIdx.y) * GM_BM, j0 = int64_t(blockIdx.x) * GM_BN;
  if (lower_only && j0 > i0) return;
  const int64_t b = blockIdx.z;
  A += b * sA;
  B += b * sB;
  C += b * sC;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  float ra[LPT], rb[LPT];
  auto gload = [&](int64_t t0) {
#pragma unroll
    for (int k = 0; k < LPT; ++k) {
      const int e = tid + 256 * k;
      int t, i;
      if (AT) {
        t = e / GM_BM;
        i = e % GM_BM;
      } else {
        i = e / GM_BK;
        t = e % GM_BK;
      }
      const int64_t gi = i0 + i, gt = t0 + t;
      ra[k] = (gi < M && gt < Kc) ? (AT ? A[gt * lda + gi] : A[gi * lda + gt]) : 0.f;
      const int tb = e / GM_BN, jb = e % GM_BN;
      const int64_t gj = j0 + jb, gtb = t0 + tb;
      rb[k] = (gj < N && gtb < Kc) ? B[gtb * ldb + gj] : 0.f;
    }
  };
  auto sstore = [&](int buf) {
#pragma unroll
    for (int k = 0; k < LPT; ++k) {
      const int e = tid + 256 * k;
      if (AT)
        As[buf][e / GM_BM][e % GM_BM] = ra[k];
      else
        As[buf][e % GM_BK][e / GM_BK] = ra[k];
      Bs[buf][e / GM_BN][e % GM_BN] = rb[k];
    }
  };
  double acc[4][4];
  float run_sum[4][4];
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      acc[p][q] = 0.0;
      run_sum[p][q] = 0.f;
    }
  gload(0);
  sstore(0);
  __syncthreads();
  int run = 0, buf = 0;
  for (int64_t t0 = 0; t0 < Kc; t0 += GM_BK) {
    const bool more = t0 + GM_BK < Kc;
    if (more) gload(t0 + GM_BK);
    float part[4][4];
#pragma unroll
    for (int p = 0; p < 4; ++p)
#pragma unroll
      for (int q = 0; q < 4; ++q) part[p][q] = 0.f;
#pragma unroll
    for (int t = 0; t < GM_BK; ++t) {
      const float4 a4 = *reinterpret_cast<const float4*>(&As[buf][t][ty * 4]);
      const float4 b4 = *reinterpret_cast<const float4*>(&Bs[buf][t][tx * 4]);
      const float av[4] = {a4.x, a4.y, a4.z, a4.w};
      const float bv[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) part[p][q] = fmaf(av[p], bv[q], part[p][q]);
    }
    if (more) sstore(buf ^ 1);
    __syncthreads();
    buf ^= 1;
#pragma unroll
    for (int p = 0; p < 4; ++p)
#pragma unroll
      for (int q = 0; q < 4; ++q) run_sum[p][q] += part[p][q];
    if (++run == GM_RUN) {
      run = 0;
#pragma unroll
      for (int p = 0; p < 4; ++p)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          acc[p][q] += double(run_sum[p][q]);
          run_sum[p][q] = 0.f;
        }
    }
  }
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t gi = i0 + ty * 4 + p, gj = j0 + tx * 4 + q;
      if (gi < M && gj < N && LOCA_CHECK(gi * ldc + gj, (M - 1) * ldc + N))
        C[gi * ldc + gj] = TC(acc[p][q] + double(run_sum[p][q]));
    }
}

// K (mp x mp): rows / columns >= m become the identity; beta is added to the first m diagonal
// entries.
__global__ void k_cr_pad(double* __restrict__ K, int64_t m, int64_t mp, double beta) {
  const int64_t total = mp * mp;
  for (int64_t e = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; e < total; e += int64_t(gridDim.x) * blockDim.x) {
    const int64_t i = e / mp, j = e % mp;
    if (i >= m || j >= m)
      K[e] = (i == j) ? 1.0 : 0.0;
    else if (i == j)
      K[e] += beta;
  }
}

// Load a 64 x 64 fp64 tile (row stride ld) into shared memory (row stride NBP).
__device__ __forceinline__ void load_tile(double (*S)[NBP], const double* __restrict__ src, int64_t ld) {
  for (int e = threadIdx.x; e < NB * NB; e += blockDim.x) {
    const int r = e / NB, c = e % NB;
    S[r][c] = src[int64_t(r) * ld + c];
  }
}

// Diagonal tile jb: factor in shared memory (unblocked, right-looking), write the factor back,
// and write the inverse of the triangular factor to Dinv[jb].  A pivot that is not positive
// sets the failure flag (E^T E + beta I is not positive definite in floating point).  Thread
// (ty, tx) of the 16 x 16 grid owns entries (ty + 16 p, tx + 16 q).
__global__ void __launch_bounds__(256) k_cr_potrf(double* __restrict__ K, int64_t mp, int jb,
                                                 double* __restrict__ Dinv, int32_t* flag) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  double(*S)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem);
  double(*X)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem + sizeof(double) * NB * NBP);
  __shared__ double rinv[NB];
  __shared__ int bad;
  if (failed(flag)) return;
  const int tid = threadIdx.x, tx = tid & 15, ty = tid >> 4;
  const int64_t o = int64_t(jb) * NB;
  double* Kd = K + o * mp + o;
  for (int e = tid; e < NB * NB; e += 256) {
    const int r = e / NB, c = e % NB;
    S[r][c] = (c <= r) ? Kd[int64_t(r) * mp + c] : 0.0;
    X[r][c] = (r == c) ? 1.0 : 0.0;
  }
  if (tid == 0) bad = 0;
  __syncthreads();
  for (int c = 0; c < NB; ++c) {
    const double piv = S[c][c];
    if (!(piv > 0.0)) {
      bad = 1;
      break;
    }
    const double lc = sqrt(piv);
    const double inv = 1.0 / lc;
    __syncthreads();
    if (tid < NB) {
      if (tid > c) S[tid][c] *= inv;
      if (tid == c) {
        S[c][c] = lc;
        rinv[c] = inv;
      }
    }
    __syncthreads();
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const int rr = ty + 16 * p;
      if (rr <= c) continue;
      const double lrc = S[rr][c];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int ss = tx + 16 * q;
        if (ss > c && ss <= rr) S[rr][ss] = fma(-lrc, S[ss][c], S[rr][ss]);
      }
    }
    __syncthreads();
  }
  if (bad) {
    if (tid == 0) atomicExch(flag, 1);
    return;
  }
  for (int e = tid; e < NB * NB; e += 256) {
    const int r = e / NB, c = e % NB;
    if (c <= r) Kd[int64_t(r) * mp + c] = S[r][c];
  }
  // X = L^-1, right-looking on the identity: row c scaled by 1 / L_cc, then removed from the rows
  // below
  for (int c = 0; c < NB; ++c) {
    if (tid <= c) X[c][tid] *= rinv[c];
    __syncthreads();
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const int rr = ty + 16 * p;
      if (rr <= c) continue;
      const double lrc = S[rr][c];
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int u = tx + 16 * q;
        if (u <= c) X[rr][u] = fma(-lrc, X[c][u], X[rr][u]);
      }
    }
    __syncthreads();
  }
  double* D = Dinv + int64_t(jb) * NB * NB;
  for (int e = tid; e < NB * NB; e += 256) D[e] = X[e / NB][e % NB];
}

// Panel: L(ib, jb) = A(ib, jb) L(jb, jb)^-T for ib = jb + 1 + blockIdx.x.
__global__ void __launch_bounds__(256) k_cr_trsm(double* __restrict__ K, int64_t mp, int jb,
                                                const double* __restrict__ Dinv, const int32_t* flag) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  double(*At)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem);
  double(*Dt)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem + sizeof(double) * NB * NBP);
  if (failed(flag)) return;
  const int ib = jb + 1 + blockIdx.x;
  double* Ab = K + int64_t(ib) * NB * mp + int64_t(jb) * NB;
  load_tile(At, Ab, mp);
  load_tile(Dt, Dinv + int64_t(jb) * NB * NB, NB);
  __syncthreads();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  double acc[4][4] = {};
  for (int u = 0; u < NB; ++u) {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const double a = At[ty + 16 * p][u];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[p][q] = fma(a, Dt[tx + 16 * q][u], acc[p][q]);
    }
  }
  __syncthreads();
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) Ab[int64_t(ty + 16 * p) * mp + tx + 16 * q] = acc[p][q];
}

// Trailing update: A(ib, kb) -= L(ib, jb) L(kb, jb)^T for jb < kb <= ib (one tile per CTA).
__global__ void __launch_bounds__(256) k_cr_syrk(double* __restrict__ K, int64_t mp, int jb, const int32_t* flag) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  double(*Li)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem);
  double(*Lk)[NBP] = reinterpret_cast<double(*)[NBP]>(cr_smem + sizeof(double) * NB * NBP);
  if (failed(flag)) return;
  const int x = blockIdx.x;
  int ii = int((sqrt(8.0 * x + 1.0) - 1.0) * 0.5);
  while ((ii + 1) * (ii + 2) / 2 <= x) ++ii;
  while (ii * (ii + 1) / 2 > x) --ii;
  const int kk = x - ii * (ii + 1) / 2;
  const int ib = jb + 1 + ii, kb = jb + 1 + kk;
  load_tile(Li, K + int64_t(ib) * NB * mp + int64_t(jb) * NB, mp);
  load_tile(Lk, K + int64_t(kb) * NB * mp + int64_t(jb) * NB, mp);
  __syncthreads();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  double acc[4][4] = {};
  for (int u = 0; u < NB; ++u) {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const double a = Li[ty + 16 * p][u];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[p][q] = fma(a, Lk[tx + 16 * q][u], acc[p][q]);
    }
  }
  double* Cb = K + int64_t(ib) * NB * mp + int64_t(kb) * NB;
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int64_t o = int64_t(ty + 16 * p) * mp + tx + 16 * q;
      Cb[o] -= acc[p][q];
    }
}

// Blocked substitution on W (mp x n, in place; T = double or float), one step per launch, on
// column tiles of TW columns (blockIdx.y):
//   MODE 0  forward diagonal:  W_ib = L(ib, ib)^-1 W_ib
//   MODE 1  forward update:    W_tb -= L(tb, ib) W_ib,    tb = ib + 1 + blockIdx.x
//   MODE 2  backward diagonal: W_ib = L(ib, ib)^-T W_ib
//   MODE 3  backward update:   W_tb -= L(ib, tb)^T W_ib,  tb = blockIdx.x < ib
template <typename T, int MODE, int TW>
__global__ void __launch_bounds__(256) k_cr_tsolve(const T* __restrict__ K, int64_t mp, const T* __restrict__ Dinv,
                                                  T* __restrict__ W, int64_t n, int ib, const int32_t* flag) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  T(*Mt)[NBP] = reinterpret_cast<T(*)[NBP]>(cr_smem);
  T(*Rt)[NBP] = reinterpret_cast<T(*)[NBP]>(cr_smem + sizeof(T) * NB * NBP);
  if (failed(flag)) return;
  constexpr bool kTrans = (MODE >= 2);
  constexpr bool kSub = (MODE == 1 || MODE == 3);
  constexpr int QN = TW / 16;
  int tb;
  const T* mat;
  int64_t ldm;
  if (MODE == 0 || MODE == 2) {
    tb = ib;
    mat = Dinv + int64_t(ib) * NB * NB;
    ldm = NB;
  } else if (MODE == 1) {
    tb = ib + 1 + blockIdx.x;
    mat = K + int64_t(tb) * NB * mp + int64_t(ib) * NB;
    ldm = mp;
  } else {
    tb = blockIdx.x;
    mat = K + int64_t(ib) * NB * mp + int64_t(tb) * NB;
    ldm = mp;
  }
  const int64_t c0 = int64_t(blockIdx.y) * TW;
  for (int e = threadIdx.x; e < NB * NB; e += 256) Mt[e / NB][e % NB] = mat[int64_t(e / NB) * ldm + e % NB];
  for (int e = threadIdx.x; e < NB * TW; e += 256) {
    const int u = e / TW, c = e % TW;
    Rt[u][c] = (c0 + c < n) ? W[(int64_t(ib) * NB + u) * n + c0 + c] : T(0);
  }
  __syncthreads();
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  T acc[4][QN];
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < QN; ++q) acc[p][q] = T(0);
  for (int u = 0; u < NB; ++u) {
#pragma unroll
    for (int p = 0; p < 4; ++p) {
      const int r = ty + 16 * p;
      const T a = kTrans ? Mt[u][r] : Mt[r][u];
#pragma unroll
      for (int q = 0; q < QN; ++q) acc[p][q] = fma(a, Rt[u][tx + 16 * q], acc[p][q]);
    }
  }
  __syncthreads();
#pragma unroll
  for (int p = 0; p < 4; ++p)
#pragma unroll
    for (int q = 0; q < QN; ++q) {
      const int64_t c = c0 + tx + 16 * q;
      if (c >= n) continue;
      T* dst = W + (int64_t(tb) * NB + ty + 16 * p) * n + c;
      *dst = kSub ? (*dst - acc[p][q]) : acc[p][q];
    }
}

template <typename TI, typename TO>
__global__ void k_cr_cvt(const TI* __restrict__ x, TO* __restrict__ y, int64_t count) {
  for (int64_t e = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; e < count; e += int64_t(gridDim.x) * blockDim.x)
    y[e] = TO(x[e]);
}

constexpr int QR_STAGE = 64;   // rows staged at a time by k_cr_vtv
constexpr int QR_CHUNK = 256;  // rows per CTA of k_cr_vtv / k_cr_qr_apply

// Partial Gram matrices of block l's ell columns of V (rows x n, columns l ell ..):
// part[l][chunk] (ELLP x ELLP, zero outside ell x ell) = sum over the chunk's rows of v v^T.
template <int ELLP>
__global__ void __launch_bounds__(256) k_cr_vtv(const double* __restrict__ V, int64_t rows, int64_t n, int ell,
                                               int nch, double* __restrict__ part) {
  __shared__ double Vs[QR_STAGE][ELLP + 1];
  constexpr int EPT = (ELLP * ELLP + 255) / 256;
  const int ch = blockIdx.x, l = blockIdx.y, tid = threadIdx.x;
  const int64_t r0 = int64_t(ch) * QR_CHUNK;
  const int64_t r1 = (r0 + QR_CHUNK < rows) ? r0 + QR_CHUNK : rows;
  double acc[EPT];
#pragma unroll
  for (int k = 0; k < EPT; ++k) acc[k] = 0.0;
  for (int64_t rs = r0; rs < r1; rs += QR_STAGE) {
    __syncthreads();
    for (int e = tid; e < QR_STAGE * ELLP; e += 256) {
      const int rr = e / ELLP, c = e % ELLP;
      Vs[rr][c] = (rs + rr < r1 && c < ell) ? V[(rs + rr) * n + int64_t(l) * ell + c] : 0.0;
    }
    __syncthreads();
#pragma unroll
    for (int k = 0; k < EPT; ++k) {
      const int e = tid + 256 * k;
      if (e < ELLP * ELLP) {
        const int a = e / ELLP, b = e % ELLP;
        double sacc = acc[k];
        for (int rr = 0; rr < QR_STAGE; ++rr) sacc = fma(Vs[rr][a], Vs[rr][b], sacc);
        acc[k] = sacc;
      }
    }
  }
  double* out = part + (int64_t(l) * nch + ch) * ELLP * ELLP;
#pragma unroll
  for (int k = 0; k < EPT; ++k) {
    const int e = tid + 256 * k;
    if (e < ELLP * ELLP) out[e] = acc[k];
  }
}

// Per block: S = sum of the partials (fixed order), S = Lc Lc^T by Cholesky (warp 0) with
// dependent columns (new component below 1e-7 of the column's norm: pivot <= 1e-14 S_cc) given
// a zero column in Lc.  Writes Lc with its diagonal replaced by the reciprocals (0 when
// dependent) to fac[l] (ELLP x ELLP).
template <int ELLP>
__global__ void __launch_bounds__(256) k_cr_qr_factor(const double* __restrict__ part, int nch, int ell,
                                                     double* __restrict__ fac) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  double(*S)[ELLP + 1] = reinterpret_cast<double(*)[ELLP + 1]>(cr_smem);
  double(*Lc)[ELLP + 1] = reinterpret_cast<double(*)[ELLP + 1]>(cr_smem + sizeof(double) * ELLP * (ELLP + 1));
  const int l = blockIdx.x, tid = threadIdx.x;
  for (int e = tid; e < ELLP * ELLP; e += blockDim.x) {
    double v = 0.0;
    for (int ch = 0; ch < nch; ++ch) v += part[(int64_t(l) * nch + ch) * ELLP * ELLP + e];
    S[e / ELLP][e % ELLP] = v;
    Lc[e / ELLP][e % ELLP] = 0.0;
  }
  __syncthreads();
  if (tid < 32) {
    const int lane = tid;
    for (int c = 0; c < ell; ++c) {
      double dsum = S[c][c];
      for (int u = 0; u < c; ++u) dsum -= Lc[c][u] * Lc[c][u];
      const bool dep = !(S[c][c] > 0.0) || !(dsum > 1e-14 * S[c][c]);
      const double lcc = dep ? 0.0 : sqrt(dsum);
      __syncwarp();
      for (int j = c + 1 + lane; j < ell; j += 32) {
        double v = 0.0;
        if (!dep) {
          v = S[j][c];
          for (int u = 0; u < c; ++u) v -= Lc[j][u] * Lc[c][u];
          v /= lcc;
        }
        Lc[j][c] = v;
      }
      if (lane == 0) Lc[c][c] = lcc;
      __syncwarp();
    }
  }
  __syncthreads();
  double* F = fac + int64_t(l) * ELLP * ELLP;
  for (int e = tid; e < ELLP * ELLP; e += blockDim.x) {
    const int a = e / ELLP, b = e % ELLP;
    double v = (b < a) ? Lc[a][b] : 0.0;
    if (a == b) v = (Lc[a][a] > 0.0) ? 1.0 / Lc[a][a] : 0.0;
    F[e] = v;
  }
}

// Per row v of block l's columns: q = v R^-1 with R = Lc^T, i.e. Lc q^T = v^T by forward
// substitution (dependent columns give q_c = 0).
template <int ELLP>
__global__ void __launch_bounds__(QR_CHUNK) k_cr_qr_apply(double* __restrict__ V, int64_t rows, int64_t n, int ell,
                                                         const double* __restrict__ fac) {
  __shared__ double F[ELLP][ELLP + 1];
  const int l = blockIdx.y, tid = threadIdx.x;
  for (int e = tid; e < ELLP * ELLP; e += QR_CHUNK) F[e / ELLP][e % ELLP] = fac[int64_t(l) * ELLP * ELLP + e];
  __syncthreads();
  const int64_t rrow = int64_t(blockIdx.x) * QR_CHUNK + tid;
  if (rrow >= rows || !LOCA_CHECK_SPAN(rrow * n + int64_t(l) * ell, ell, rows * n)) return;
  double* v = V + rrow * n + int64_t(l) * ell;
  double x[ELLP];
#pragma unroll
  for (int c = 0; c < ELLP; ++c) x[c] = (c < ell) ? v[c] : 0.0;
#pragma unroll
  for (int c = 0; c < ELLP; ++c) {
    double a = x[c];
#pragma unroll
    for (int u = 0; u < c; ++u) a = fma(-F[c][u], x[u], a);
    x[c] = a * F[c][c];
  }
#pragma unroll
  for (int c = 0; c < ELLP; ++c)
    if (c < ell) v[c] = x[c];
}

// Partial Gram matrices of B^T (d x ell per block): part[l][chunk][a][b] = sum over the chunk's
// rows of Bt[j][a] Bt[j][b].
__global__ void __launch_bounds__(256) k_cr_btb(const double* __restrict__ Bt, int64_t d, int64_t n, int ell,
                                               int nch, double* __restrict__ part) {
  const int ch = blockIdx.x, l = blockIdx.y;
  const double* Bb = Bt + int64_t(l) * ell;
  const int64_t j0 = int64_t(ch) * RZ_CH;
  const int64_t j1 = (j0 + RZ_CH < d) ? j0 + RZ_CH : d;
  double* out = part + (int64_t(l) * nch + ch) * ell * ell;
  for (int e = threadIdx.x; e < ell * ell; e += blockDim.x) {
    const int a = e / ell, b = e % ell;
    double s = 0.0;
    for (int64_t j = j0; j < j1; ++j) s = fma(Bb[j * n + a], Bb[j * n + b], s);
    out[e] = s;
  }
}

// Per block: B B^T from the partials (fixed order), its eigen-decomposition, and the leading r
// eigenpairs: Ur[l] (ell x r, eigenvectors as columns) and sig[l] (r singular values).
template <int ELLP>
__global__ void __launch_bounds__(256) k_cr_ritz_eig(const double* __restrict__ part, int nch, int ell, int r,
                                                    const int32_t* flag, int32_t* status, double* __restrict__ Ur,
                                                    double* __restrict__ sig, float* __restrict__ sigma_out) {
  extern __shared__ __align__(16) unsigned char cr_smem[];
  double(*A)[ELLP] = reinterpret_cast<double(*)[ELLP]>(cr_smem);
  double(*V)[ELLP] = reinterpret_cast<double(*)[ELLP]>(cr_smem + sizeof(double) * ELLP * ELLP);
  int* order = reinterpret_cast<int*>(cr_smem + 2 * sizeof(double) * ELLP * ELLP);
  const int l = blockIdx.x, tid = threadIdx.x;
  double* Ul = Ur + int64_t(l) * ell * r;
  double* sl = sig + int64_t(l) * r;
  if (failed(flag)) {
    if (tid == 0 && l == 0) atomicExch(status, int32_t(LOCA_ERR_NUMERIC));
    for (int e = tid; e < ell * r; e += blockDim.x) Ul[e] = 0.0;
    for (int e = tid; e < r; e += blockDim.x) {
      sl[e] = 0.0;
      if (sigma_out != nullptr) sigma_out[int64_t(l) * r + e] = 0.f;
    }
    return;
  }
  for (int e = tid; e < ELLP * ELLP; e += blockDim.x) {
    const int a = e / ELLP, b = e % ELLP;
    double s = 0.0;
    if (a < ell && b < ell)
      for (int ch = 0; ch < nch; ++ch) s += part[((int64_t(l) * nch + ch) * ell + a) * ell + b];
    A[a][b] = s;
    V[a][b] = (a == b) ? 1.0 : 0.0;
  }
  __syncthreads();
  // symmetrise (the two triangles are summed in the same order, so this only removes nothing
  // but rounding asymmetry from the fma chains)
  for (int e = tid; e < ELLP * ELLP; e += blockDim.x) {
    const int a = e / ELLP, b = e % ELLP;
    if (a > b) A[a][b] = A[b][a];
  }
  __syncthreads();
  jacobi_eig_block<ELLP>(A, V, order, ell);
  __syncthreads();
  const double lam1 = A[order[0]][order[0]];
  const double s1 = lam1 > 0.0 ? sqrt(lam1) : 0.0;
  for (int i = tid; i < r; i += blockDim.x) {
    const double lam = A[order[i]][order[i]];
    double sg = lam > 0.0 ? sqrt(lam) : 0.0;
    if (!(sg > 1e-12 * s1)) sg = 0.0;
    sl[i] = sg;
    if (sigma_out != nullptr) sigma_out[int64_t(l) * r + i] = float(sg);
  }
  for (int e = tid; e < ell * r; e += blockDim.x) {
    const int c = e / r, i = e % r;
    Ul[e] = V[c][order[i]];
  }
}

// P_l[a][i] = sigma_i (Q_Y U_B)[a][i] for the chunk's rows a < m, and Q_l[i][j] =
// (B^T U_B)[j][i] / sigma_i for the chunk's columns j < d, with each chunk's entry of largest
// magnitude per Q_l row (value, lowest index on ties) for the sign convention.
__global__ void __launch_bounds__(RZ_CH) k_cr_ritz_out(const double* __restrict__ QY, const double* __restrict__ Bt,
                                                      int64_t n, int64_t m, int64_t d, int ell, int r, int nch,
                                                      const double* __restrict__ Ur, const double* __restrict__ sig,
                                                      float* __restrict__ P, float* __restrict__ Q,
                                                      double* __restrict__ amax_v, int64_t* __restrict__ amax_i) {
  __shared__ double Us[kMaxEll * kMaxEll];
  __shared__ double ss[kMaxEll];
  __shared__ double bv[RZ_CH / 32];
  __shared__ int64_t bi[RZ_CH / 32];
  const int ch = blockIdx.x, l = blockIdx.y, tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
  for (int e = tid; e < ell * r; e += RZ_CH) Us[e] = Ur[int64_t(l) * ell * r + e];
  for (int e = tid; e < r; e += RZ_CH) ss[e] = sig[int64_t(l) * r + e];
  __syncthreads();
  const int64_t a = int64_t(ch) * RZ_CH + tid;
  if (a < m) {
    const double* row = QY + a * n + int64_t(l) * ell;
    for (int i = 0; i < r; ++i) {
      double s = 0.0;
      for (int c = 0; c < ell; ++c) s = fma(row[c], Us[c * r + i], s);
      if (LOCA_CHECK((int64_t(l) * m + a) * r + i, int64_t(gridDim.y) * m * r))
        P[(int64_t(l) * m + a) * r + i] = (ss[i] > 0.0) ? float(ss[i] * s) : 0.f;
    }
  }
  const int64_t j = int64_t(ch) * RZ_CH + tid;
  const double* brow = Bt + j * n + int64_t(l) * ell;
  for (int i = 0; i < r; ++i) {
    double v = 0.0;
    if (j < d && ss[i] > 0.0) {
      for (int c = 0; c < ell; ++c) v = fma(brow[c], Us[c * r + i], v);
      v /= ss[i];
    }
    if (j < d && LOCA_CHECK((int64_t(l) * r + i) * d + j, int64_t(gridDim.y) * r * d))
      Q[(int64_t(l) * r + i) * d + j] = float(v);
    double best = (j < d && v == v) ? fabs(v) : -1.0;  // NaN entries never win
    int64_t bj = j;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const double ob = __shfl_xor_sync(0xffffffffu, best, off);
      const int64_t oj = __shfl_xor_sync(0xffffffffu, bj, off);
      if (ob > best || (ob == best && oj < bj)) {
        best = ob;
        bj = oj;
      }
    }
    if (lane == 0) {
      bv[wid] = best;
      bi[wid] = bj;
    }
    __syncthreads();
    if (tid == 0 && LOCA_CHECK((int64_t(l) * r + i) * nch + ch, int64_t(gridDim.y) * r * nch)) {
      double b0 = bv[0];
      int64_t i0 = bi[0];
      for (int w = 1; w < RZ_CH / 32; ++w)
        if (bv[w] > b0 || (bv[w] == b0 && bi[w] < i0)) {
          b0 = bv[w];
          i0 = bi[w];
        }
      amax_v[(int64_t(l) * r + i) * nch + ch] = b0;
      amax_i[(int64_t(l) * r + i) * nch + ch] = i0;
    }
    __syncthreads();
  }
}

// Sign convention: the entry of largest magnitude of Q_l row i (lowest index on ties) is made
// positive, flipping that row and column i of P_l.  grid (L, r).
__global__ void __launch_bounds__(256) k_cr_ritz_sign(float* __restrict__ P, float* __restrict__ Q, int64_t m,
                                                     int64_t d, int r, int nch, const double* __restrict__ amax_v,
                                                     const int64_t* __restrict__ amax_i) {
  __shared__ int s_flip;
  const int l = blockIdx.x, i = blockIdx.y;
  if (threadIdx.x == 0) {
    const double* bv = amax_v + (int64_t(l) * r + i) * nch;
    const int64_t* bi = amax_i + (int64_t(l) * r + i) * nch;
    double b0 = bv[0];
    int64_t j0 = bi[0];
    for (int c = 1; c < nch; ++c)
      if (bv[c] > b0 || (bv[c] == b0 && bi[c] < j0)) {
        b0 = bv[c];
        j0 = bi[c];
      }
    s_flip = (j0 >= 0 && j0 < d && Q[(int64_t(l) * r + i) * d + j0] < 0.f) ? 1 : 0;
  }
  __syncthreads();
  if (!s_flip || !LOCA_CHECK_SPAN((int64_t(l) * r + i) * d, d, int64_t(gridDim.x) * r * d)) return;
  for (int64_t j = threadIdx.x; j < d; j += blockDim.x) Q[(int64_t(l) * r + i) * d + j] *= -1.f;
  for (int64_t a = threadIdx.x; a < m; a += blockDim.x) P[(int64_t(l) * m + a) * r + i] *= -1.f;
}

struct RsvdWs {
  size_t K, Dinv, Kf, Dinvf, Ym, Wm, Wf, Zd, Zf, Tn, qrpart, qrfac, part, Ur, sig, amv, ami, flag, total;
};

RsvdWs rsvd_ws(int64_t Np, int64_t m, int64_t d, int L, int ell, int r) {
  const int64_t mp = (m + NB - 1) / NB * NB;
  const int64_t nb = mp / NB;
  const int64_t n = int64_t(L) * ell;
  const int64_t nchd = (d + RZ_CH - 1) / RZ_CH;
  const int64_t nchq = ((m > d ? m : d) + RZ_CH - 1) / RZ_CH;
  RsvdWs w{};
  size_t o = 0;
  auto take = [&](size_t bytes) {
    const size_t at = o;
    o += align256(bytes);
    return at;
  };
  const int64_t ellp = ell <= 16 ? 16 : (ell <= 32 ? 32 : 64);
  const int64_t nchqr = ((m > d ? m : d) + QR_CHUNK - 1) / QR_CHUNK;
  w.K = take(sizeof(double) * mp * mp);
  w.Dinv = take(sizeof(double) * nb * NB * NB);
  w.Kf = take(sizeof(float) * mp * mp);
  w.Dinvf = take(sizeof(float) * nb * NB * NB);
  w.Ym = take(sizeof(double) * mp * n);
  w.Wm = take(sizeof(double) * mp * n);
  w.Wf = take(sizeof(float) * mp * n);
  w.Zd = take(sizeof(double) * d * n);
  w.Zf = take(sizeof(float) * d * n);
  w.Tn = take(sizeof(float) * Np * n);
  w.qrpart = take(sizeof(double) * L * nchqr * ellp * ellp);
  w.qrfac = take(sizeof(double) * L * ellp * ellp);
  w.part = take(sizeof(double) * L * nchd * ell * ell);
  w.Ur = take(sizeof(double) * L * ell * r);
  w.sig = take(sizeof(double) * L * r);
  w.amv = take(sizeof(double) * L * r * nchq);
  w.ami = take(sizeof(int64_t) * L * r * nchq);
  w.flag = take(sizeof(int32_t) * 64);
  w.total = o;
  return w;
}

template <bool AT, typename TC>
cudaError_t gemm(const float* A, int64_t lda, int64_t sA, const float* B, int64_t ldb, int64_t sB, TC* C,
                 int64_t ldc, int64_t sC, int64_t M, int64_t N, int64_t Kc, int batch, int lower_only,
                 cudaStream_t s) {
  const dim3 grid(unsigned((N + GM_BN - 1) / GM_BN), unsigned((M + GM_BM - 1) / GM_BM), unsigned(batch));
  k_cr_gemm<AT, TC><<<grid, 256, 0, s>>>(A, lda, sA, B, ldb, sB, C, ldc, sC, M, N, Kc, lower_only);
  return cudaGetLastError();
}

// W (mp x n) <- K^-1 W with K = L L^T (forward, then backward substitution), in T.
template <typename T>
cudaError_t solve(const T* K, int64_t mp, const T* Dinv, T* W, int64_t n, const int32_t* flag, cudaStream_t s) {
  const int nb = int(mp / NB);
  const size_t smem = sizeof(T) * 2 * NB * NBP;
  const unsigned ct16 = unsigned((n + 15) / 16), ct64 = unsigned((n + 63) / 64);
  for (int ib = 0; ib < nb; ++ib) {
    k_cr_tsolve<T, 0, 16><<<dim3(1, ct16), 256, smem, s>>>(K, mp, Dinv, W, n, ib, flag);
    if (ib + 1 < nb)
      k_cr_tsolve<T, 1, 64><<<dim3(unsigned(nb - 1 - ib), ct64), 256, smem, s>>>(K, mp, Dinv, W, n, ib, flag);
  }
  for (int ib = nb - 1; ib >= 0; --ib) {
    k_cr_tsolve<T, 2, 16><<<dim3(1, ct16), 256, smem, s>>>(K, mp, Dinv, W, n, ib, flag);
    if (ib > 0) k_cr_tsolve<T, 3, 64><<<dim3(unsigned(ib), ct64), 256, smem, s>>>(K, mp, Dinv, W, n, ib, flag);
  }
  return cudaGetLastError();
}

template <typename TI, typename TO>
cudaError_t cvt(const TI* x, TO* y, int64_t count, cudaStream_t s) {
  k_cr_cvt<TI, TO><<<2 * sm_count(), 256, 0, s>>>(x, y, count);
  return cudaGetLastError();
}

// Orthonormal basis of every block's ell columns of V (rows x n), in place: Cholesky QR twice.
template <int ELLP>
cudaError_t orth(double* V, int64_t rows, int64_t n, int ell, int L, double* qrpart, double* qrfac, cudaStream_t s) {
  const int nch = int((rows + QR_CHUNK - 1) / QR_CHUNK);
  const size_t fsmem = 2 * sizeof(double) * ELLP * (ELLP + 1);
  for (int pass = 0; pass < 2; ++pass) {
    k_cr_vtv<ELLP><<<dim3(unsigned(nch), unsigned(L)), 256, 0, s>>>(V, rows, n, ell, nch, qrpart);
    k_cr_qr_factor<ELLP><<<L, 256, fsmem, s>>>(qrpart, nch, ell, qrfac);
    k_cr_qr_apply<ELLP><<<dim3(unsigned(nch), unsigned(L)), QR_CHUNK, 0, s>>>(V, rows, n, ell, qrfac);
  }
  return cudaGetLastError();
}

cudaError_t set_smem_attributes() {
  static const void* fns64[] = {
      reinterpret_cast<const void*>(k_cr_potrf), reinterpret_cast<const void*>(k_cr_trsm),
      reinterpret_cast<const void*>(k_cr_syrk), reinterpret_cast<const void*>(k_cr_tsolve<double, 0, 16>),
      reinterpret_cast<const void*>(k_cr_tsolve<double, 1, 64>),
      reinterpret_cast<const void*>(k_cr_tsolve<double, 2, 16>),
      reinterpret_cast<const void*>(k_cr_tsolve<double, 3, 64>)};
  for (const void* f : fns64) {
    cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kTileSmem));
    if (e != cudaSuccess) return e;
  }
  static const void* fqr[] = {reinterpret_cast<const void*>(k_cr_qr_factor<16>),
                              reinterpret_cast<const void*>(k_cr_qr_factor<32>),
                              reinterpret_cast<const void*>(k_cr_qr_factor<64>)};
  for (const void* f : fqr) {
    cudaError_t e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         int(2 * sizeof(double) * 64 * 65));
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

template <int ELLP>
cudaError_t rsvd_t(const float* E, const float* G, int64_t Np, int64_t m, int64_t d, int L, float beta, int r,
                   int ell, int q, const float* Omega, float* P, float* Q, float* sigma, char* ws, int32_t* status,
                   cudaStream_t s) {
  const RsvdWs w = rsvd_ws(Np, m, d, L, ell, r);
  const int64_t mp = (m + NB - 1) / NB * NB;
  const int nb = int(mp / NB);
  const int64_t n = int64_t(L) * ell;
  double* K = reinterpret_cast<double*>(ws + w.K);
  double* Dinv = reinterpret_cast<double*>(ws + w.Dinv);
  float* Kf = reinterpret_cast<float*>(ws + w.Kf);
  float* Dinvf = reinterpret_cast<float*>(ws + w.Dinvf);
  double* Ym = reinterpret_cast<double*>(ws + w.Ym);
  double* Wm = reinterpret_cast<double*>(ws + w.Wm);
  float* Wf = reinterpret_cast<float*>(ws + w.Wf);
  double* Zd = reinterpret_cast<double*>(ws + w.Zd);
  float* Zf = reinterpret_cast<float*>(ws + w.Zf);
  float* Tn = reinterpret_cast<float*>(ws + w.Tn);
  double* qrpart = reinterpret_cast<double*>(ws + w.qrpart);
  double* qrfac = reinterpret_cast<double*>(ws + w.qrfac);
  int32_t* flag = reinterpret_cast<int32_t*>(ws + w.flag);
  cudaError_t e = set_smem_attributes();
  if (e != cudaSuccess) return e;
#define CR_TRY(x)              \
  do {                         \
    cudaError_t e_ = (x);      \
    if (e_ != cudaSuccess) return e_; \
  } while (0)
  CR_TRY(cudaMemsetAsync(flag, 0, sizeof(int32_t) * 64, s));
  CR_TRY(cudaMemsetAsync(Ym, 0, sizeof(double) * mp * n, s));
  // K = E^T E (lower tiles), + beta I, padded
  CR_TRY((gemm<true, double>(E, m, 0, E, m, 0, K, mp, 0, m, m, Np, 1, 1, s)));
  k_cr_pad<<<4 * sm_count(), 256, 0, s>>>(K, m, mp, double(beta));
  CR_TRY(cudaGetLastError());
  for (int jb = 0; jb < nb; ++jb) {
    k_cr_potrf<<<1, 256, kTileSmem, s>>>(K, mp, jb, Dinv, flag);
    const int T = nb - jb - 1;
    if (T > 0) {
      k_cr_trsm<<<T, 256, kTileSmem, s>>>(K, mp, jb, Dinv, flag);
      k_cr_syrk<<<T * (T + 1) / 2, 256, kTileSmem, s>>>(K, mp, jb, flag);
    }
    CR_TRY(cudaGetLastError());
  }
  if (q > 0) {
    CR_TRY((cvt<double, float>(K, Kf, mp * mp, s)));
    CR_TRY((cvt<double, float>(Dinv, Dinvf, int64_t(nb) * NB * NB, s)));
  }
  // Ym = F^T X for every block, X (d x ell per block, fp32) at column offset l ell of Xf (ld ldx,
  // block stride sx): Tn = G_l X, Ym = K^-1 E^T Tn (fp64 factor when exact, else the fp32 one on
  // an fp32 copy)
  auto apply_Ft = [&](const float* Xf, int64_t ldx, int64_t sx, bool exact) -> cudaError_t {
    CR_TRY((gemm<false, float>(G, d, Np * d, Xf, ldx, sx, Tn, n, ell, Np, ell, d, L, 0, s)));
    CR_TRY((gemm<true, double>(E, m, 0, Tn, n, 0, Ym, n, 0, m, n, Np, 1, 0, s)));
    if (exact) return solve<double>(K, mp, Dinv, Ym, n, flag, s);
    CR_TRY((cvt<double, float>(Ym, Wf, mp * n, s)));
    CR_TRY(solve<float>(Kf, mp, Dinvf, Wf, n, flag, s));
    return cvt<float, double>(Wf, Ym, mp * n, s);
  };
  // Zd = F Y for every block, Y = Vm (mp x n, fp64; overwritten when exact): Wf = K^-1 Y in fp32,
  // Tn = E Wf, Zd = G_l^T Tn
  auto apply_F = [&](double* Vm, bool exact) -> cudaError_t {
    if (exact) {
      CR_TRY(solve<double>(K, mp, Dinv, Vm, n, flag, s));
      CR_TRY((cvt<double, float>(Vm, Wf, mp * n, s)));
    } else {
      CR_TRY((cvt<double, float>(Vm, Wf, mp * n, s)));
      CR_TRY(solve<float>(Kf, mp, Dinvf, Wf, n, flag, s));
    }
    CR_TRY((gemm<false, float>(E, m, 0, Wf, n, 0, Tn, n, 0, Np, n, m, 1, 0, s)));
    return gemm<true, double>(G, d, Np * d, Tn, n, ell, Zd, n, ell, d, ell, Np, L, 0, s);
  };
  CR_TRY(apply_Ft(Omega, int64_t(ell), int64_t(0), q == 0));
  CR_TRY(orth<ELLP>(Ym, m, n, ell, L, qrpart, qrfac, s));
  for (int it = 0; it < q; ++it) {
    CR_TRY(apply_F(Ym, false));
    CR_TRY(orth<ELLP>(Zd, d, n, ell, L, qrpart, qrfac, s));
    CR_TRY((cvt<double, float>(Zd, Zf, d * n, s)));
    CR_TRY(apply_Ft(Zf, n, int64_t(ell), it == q - 1));
    CR_TRY(orth<ELLP>(Ym, m, n, ell, L, qrpart, qrfac, s));
  }
  // Rayleigh-Ritz: B^T = F Q_Y
  CR_TRY(cudaMemcpyAsync(Wm, Ym, sizeof(double) * mp * n, cudaMemcpyDeviceToDevice, s));
  CR_TRY(apply_F(Wm, true));
  const int nchd = int((d + RZ_CH - 1) / RZ_CH);
  const int nchq = int(((m > d ? m : d) + RZ_CH - 1) / RZ_CH);
  double* part = reinterpret_cast<double*>(ws + w.part);
  double* Ur = reinterpret_cast<double*>(ws + w.Ur);
  double* sig = reinterpret_cast<double*>(ws + w.sig);
  double* amv = reinterpret_cast<double*>(ws + w.amv);
  int64_t* ami = reinterpret_cast<int64_t*>(ws + w.ami);
  k_cr_btb<<<dim3(unsigned(nchd), unsigned(L)), 256, 0, s>>>(Zd, d, n, ell, nchd, part);
  CR_TRY(cudaGetLastError());
  const size_t eig_smem = 2 * sizeof(double) * ELLP * ELLP + sizeof(int) * ELLP;
  CR_TRY(cudaFuncSetAttribute(k_cr_ritz_eig<ELLP>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(eig_smem)));
  k_cr_ritz_eig<ELLP><<<L, 256, eig_smem, s>>>(part, nchd, ell, r, flag, status, Ur, sig, sigma);
  CR_TRY(cudaGetLastError());
  k_cr_ritz_out<<<dim3(unsigned(nchq), unsigned(L)), RZ_CH, 0, s>>>(Ym, Zd, n, m, d, ell, r, nchq, Ur, sig, P, Q, amv,
                                                                      ami);
  CR_TRY(cudaGetLastError());
  k_cr_ritz_sign<<<dim3(unsigned(L), unsigned(r)), 256, 0, s>>>(P, Q, m, d, r, nchq, amv, ami);
  CR_TRY(cudaGetLastError());
#undef CR_TRY
  return cudaSuccess;
}

}  // namespace

int calib_rsvd_max_ell() { return kMaxEll; }
int64_t calib_rsvd_max_width() { return kMaxWidth; }

size_t calib_rsvd_workspace_bytes(int64_t Np, int64_t m, int64_t d, int L, int ell, int r) {
  return rsvd_ws(Np, m, d, L, ell, r).total;
}

cudaError_t launch_calib_rsvd(const float* E_probe, const float* G_probe, int64_t Np, int64_t m, int64_t d, int L,
                              float beta, int r, int ell, int q, const float* Omega, float* P, float* Q,
                              float* sigma, void* workspace, int32_t* status, cudaStream_t s) {
  char* ws = static_cast<char*>(workspace);
  if (ell <= 16) return rsvd_t<16>(E_probe, G_probe, Np, m, d, L, beta, r, ell, q, Omega, P, Q, sigma, ws, status, s);
  if (ell <= 32) return rsvd_t<32>(E_probe, G_probe, Np, m, d, L, beta, r, ell, q, Omega, P, Q, sigma, ws, status, s);
  return rsvd_t<64>(E_probe, G_probe, Np, m, d, L, beta, r, ell, q, Omega, P, Q, sigma, ws, status, s);
}

}  // namespace loca
