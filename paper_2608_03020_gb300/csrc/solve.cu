// Projected statistics and batched positive-definite solves (Eqs. 8 and 9; Theorem S6; S7).
//
// k_project_rows  (shapes the tensor-core projection of project_tc.cu does not take: d or k not a
//                 multiple of 4, unaligned pointers)
//                 GA_l = Gram_l A_l, CA_l = Cross_l A_l (d x k each), as PR_SPLIT partial
//                 products over quarters of the column range (GA = sum_z GA_z, summed in a fixed
//                 order by k_chol_solve).  A CTA takes 256 rows of the stacked [Gram_l; Cross_l]
//                 and one column quarter; 32-column slabs of its rows are staged in shared memory
//                 by row-contiguous 16-byte loads (a warp request covers 4 rows, so L1 sees 4
//                 lines per request, not 32), then each thread forms a register block of
//                 RPT rows x SPT columns of the product with A's slab (broadcast reads).  Bound: the
//                 HBM read of Gram and Cross (8 d^2 bytes per block).
// k_chol_solve    one thread block per (ridge candidate j, block l):
//                 GA_l and CA_l summed over their nsplit partial products (fixed order),
//                 G_l = A_l^T GA_l (k x k), lambda from the trace, Cholesky of G_l + lambda I in
//                 fp64 in shared memory, then every row i of C_l = B_prev,l G_l + s_l CA_l
//                 (s_l = cross_scale[l], or 1) is solved
//                 by a forward and a back substitution:  B[j, l, i] = C_l[i] (G_l + lambda I)^-1.
//                 k is padded to a compile-time size with an identity block (its solution
//                 columns are zero), so each row's solve stays in registers.
#include "chol.cuh"
#include "loca_internal.h"

namespace loca {
namespace {

constexpr int PR_THREADS = 256;
constexpr int PR_ROWS = 256;   // rows per CTA
constexpr int PR_JC = 32;      // columns per staged slab
constexpr int PR_LD = PR_JC + 4;
constexpr int PR_SPLIT = 4;    // column ranges per row (partial products)

template <int KM>
__global__ void __launch_bounds__(PR_THREADS, KM <= 16 ? 3 : 1) k_project_rows(const float* __restrict__ gram,
                                                            const float* __restrict__ cross,
                                                            const float* __restrict__ A, int64_t d,
                                                            int k, float* __restrict__ GA,
                                                            float* __restrict__ CA) {
  constexpr int SPT = KM < 8 ? KM : 8;         // product columns per thread
  constexpr int G = KM / SPT;                  // column groups
  constexpr int RPT = PR_ROWS * G / PR_THREADS;  // rows per thread
  constexpr int RS = PR_ROWS / RPT;            // row stride between a thread's rows
  extern __shared__ __align__(16) float pr_smem[];
  float* Ms = pr_smem;                          // PR_ROWS x PR_LD
  float* As = pr_smem + PR_ROWS * PR_LD;        // PR_JC x KM
  const int l = blockIdx.y, z = blockIdx.z, tid = threadIdx.x;
  const int64_t zlen = ((d + PR_SPLIT * PR_JC - 1) / (PR_SPLIT * PR_JC)) * PR_JC;
  const int64_t jb = int64_t(z) * zlen;
  const int64_t je = (jb + zlen < d) ? jb + zlen : d;
  const int64_t row0 = int64_t(blockIdx.x) * PR_ROWS;  // in the stacked [Gram; Cross], 2d rows
  const float* Al = A + int64_t(l) * d * k;
  const bool vec = (d % 4 == 0);
  const int g = tid % G, rs = tid / G;
  float acc[RPT][SPT];
#pragma unroll
  for (int i = 0; i < RPT; ++i)
#pragma unroll
    for (int s = 0; s < SPT; ++s) acc[i][s] = 0.f;
  // each thread moves PR_LOADS 16-byte pieces of a slab: all are loaded into registers before any
  // is stored, and the next slab's loads are in flight while the current one is multiplied
  constexpr int PR_LOADS = PR_ROWS * (PR_JC / 4) / PR_THREADS;
  constexpr int PR_ALOADS = (PR_JC * KM + PR_THREADS - 1) / PR_THREADS;
  float4 pre[PR_LOADS];
  float apre[PR_ALOADS];
  auto gload = [&](int64_t j0) {
    const int jn = int((je - j0) < PR_JC ? (je - j0) : PR_JC);
#pragma unroll
    for (int it = 0; it < PR_ALOADS; ++it) {
      const int e = tid + it * PR_THREADS;
      const int jj = e / KM, s = e % KM;
      apre[it] = (e < PR_JC * KM && jj < jn && s < k && LOCA_CHECK((j0 + jj) * k + s, d * k))
                     ? __ldg(Al + (j0 + jj) * k + s)
                     : 0.f;
    }
#pragma unroll
    for (int it = 0; it < PR_LOADS; ++it) {
      const int e = tid + it * PR_THREADS;
      const int rr = e / (PR_JC / 4), c4 = (e % (PR_JC / 4)) * 4;
      const int64_t row = row0 + rr;
      float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
      if (row < 2 * d && LOCA_CHECK_SPAN((row < d ? row : row - d) * d + j0 + c4, c4 + 4 <= jn ? 4 : jn - c4, d * d)) {
        const float* M = (row < d ? gram + int64_t(l) * d * d + row * d
                                  : cross + int64_t(l) * d * d + (row - d) * d) + j0 + c4;
        if (vec && c4 + 4 <= jn) {
          v = __ldg(reinterpret_cast<const float4*>(M));
        } else {
          if (c4 + 0 < jn) v.x = M[0];
          if (c4 + 1 < jn) v.y = M[1];
          if (c4 + 2 < jn) v.z = M[2];
          if (c4 + 3 < jn) v.w = M[3];
        }
      }
      pre[it] = v;
    }
  };
  if (jb < je) gload(jb);
  for (int64_t j0 = jb; j0 < je; j0 += PR_JC) {
    __syncthreads();  // the previous slab's products are done with Ms and As
#pragma unroll
    for (int it = 0; it < PR_LOADS; ++it) {
      const int e = tid + it * PR_THREADS;
      *reinterpret_cast<float4*>(&Ms[(e / (PR_JC / 4)) * PR_LD + (e % (PR_JC / 4)) * 4]) = pre[it];
    }
#pragma unroll
    for (int it = 0; it < PR_ALOADS; ++it) {
      const int e = tid + it * PR_THREADS;
      if (e < PR_JC * KM) As[e] = apre[it];
    }
    __syncthreads();
    if (j0 + PR_JC < je) gload(j0 + PR_JC);
#pragma unroll 4
    for (int jj = 0; jj < PR_JC; ++jj) {
      float av[SPT];
#pragma unroll
      for (int s = 0; s < SPT; ++s) av[s] = As[jj * KM + g * SPT + s];
#pragma unroll
      for (int i = 0; i < RPT; ++i) {
        const float m = Ms[(rs + RS * i) * PR_LD + jj];
#pragma unroll
        for (int s = 0; s < SPT; ++s) acc[i][s] = fmaf(m, av[s], acc[i][s]);
      }
    }
  }
  const int64_t part = int64_t(z) * gridDim.y * d * k;
#pragma unroll
  for (int i = 0; i < RPT; ++i) {
    const int64_t row = row0 + rs + RS * i;
    if (row >= 2 * d) continue;
    const bool is_gram = row < d;
    const int64_t ri = is_gram ? row : row - d;
    float* out = (is_gram ? GA : CA) + part + (int64_t(l) * d + ri) * k;
#pragma unroll
    for (int s = 0; s < SPT; ++s)
      if (g * SPT + s < k && LOCA_CHECK(part + (int64_t(l) * d + ri) * k + g * SPT + s, int64_t(PR_SPLIT) * gridDim.y * d * k))
        out[g * SPT + s] = acc[i][s];
  }
}

constexpr int CS_THREADS = 256;
constexpr int CS_ROWS = 64;  // rows of A / GA staged per step when forming G

template <int KM>
__global__ void __launch_bounds__(CS_THREADS) k_chol_solve(
    const float* __restrict__ GA, const float* __restrict__ CA, int nsplit, const float* __restrict__ A,
    const float* __restrict__ B_prev, const double* __restrict__ xsq_total, const float* __restrict__ cross_scale,
    int64_t d, int k, int L,
    float l0, float l1, float l2, float l3, float l4, float l5, float l6, float l7, float l8,
    float l9, float l10, float l11, float l12, float l13, float l14, float l15,
    float* __restrict__ B, int32_t* __restrict__ info, float* __restrict__ G_out,
    float* __restrict__ C_out) {
  __shared__ float As[CS_ROWS][KM];
  __shared__ float Gs[CS_ROWS][KM];
  __shared__ float Gf[KM][KM];   // G_l (fp32, symmetrised), padded with identity
  __shared__ double Md[KM][KM];  // G_l + lambda I, then its Cholesky factor (lower)
  __shared__ float Lf[KM][KM];
  __shared__ float Linv[KM];
  __shared__ int s_info;
  const int j = blockIdx.x, l = blockIdx.y;
  const float lam_rel[16] = {l0, l1, l2, l3, l4, l5, l6, l7, l8, l9, l10, l11, l12, l13, l14, l15};
  const float* Al = A + int64_t(l) * d * k;
  const float* GAl = GA + int64_t(l) * d * k;
  const float* CAl = CA + int64_t(l) * d * k;
  const int64_t zs = int64_t(L) * d * k;  // stride between the nsplit partial products

  // G_l = A_l^T GA_l: thread owns entries e = t, t + 256, ... of the KM x KM matrix
  constexpr int PER = (KM * KM + CS_THREADS - 1) / CS_THREADS;
  float g[PER];
#pragma unroll
  for (int p = 0; p < PER; ++p) g[p] = 0.f;
  for (int64_t i0 = 0; i0 < d; i0 += CS_ROWS) {
    __syncthreads();
    for (int e = threadIdx.x; e < CS_ROWS * KM; e += CS_THREADS) {
      const int ii = e / KM, s = e % KM;
      const bool ok = (i0 + ii < d) && s < k && LOCA_CHECK((i0 + ii) * k + s, d * k);
      As[ii][s] = ok ? Al[(i0 + ii) * k + s] : 0.f;
      float gsum = 0.f;
      if (ok)
        for (int z = 0; z < nsplit; ++z) gsum += GAl[z * zs + (i0 + ii) * k + s];
      Gs[ii][s] = gsum;
    }
    __syncthreads();
#pragma unroll
    for (int p = 0; p < PER; ++p) {
      const int e = threadIdx.x + p * CS_THREADS;
      if (e < KM * KM) {
        const int a = e / KM, b = e % KM;
        float acc = g[p];
        for (int ii = 0; ii < CS_ROWS; ++ii) acc = fmaf(As[ii][a], Gs[ii][b], acc);
        g[p] = acc;
      }
    }
  }
#pragma unroll
  for (int p = 0; p < PER; ++p) {
    const int e = threadIdx.x + p * CS_THREADS;
    if (e < KM * KM) Gf[e / KM][e % KM] = g[p];
  }
  __syncthreads();
  const double lam =
      double(lam_rel[j]) * (xsq_total != nullptr ? xsq_total[l] / double(d) : 1.0);
  for (int e = threadIdx.x; e < KM * KM; e += CS_THREADS) {
    const int a = e / KM, b = e % KM;
    double v;
    if (a < k && b < k) {
      v = 0.5 * (double(Gf[a][b]) + double(Gf[b][a]));
      if (a == b) v += lam;
    } else {
      v = (a == b) ? 1.0 : 0.0;
    }
    Md[a][b] = v;
  }
  __syncthreads();
  if (G_out != nullptr && j == 0) {
    for (int e = threadIdx.x; e < k * k; e += CS_THREADS) {
      const int a = e / k, b = e % k;
      if (LOCA_CHECK((int64_t(l) * k + a) * k + b, int64_t(L) * k * k))
        G_out[(int64_t(l) * k + a) * k + b] = float(0.5 * (double(Gf[a][b]) + double(Gf[b][a])));
    }
  }
  const int inf = chol_factor<KM>(Md, Lf, Linv, &s_info);
  if (threadIdx.x == 0 && LOCA_CHECK(int64_t(j) * L + l, int64_t(gridDim.x) * L)) info[int64_t(j) * L + l] = inf;

  float* Bj = B + (int64_t(j) * L + l) * d * k;
  const float* Bp = B_prev ? B_prev + int64_t(l) * d * k : nullptr;
  const float cs = cross_scale != nullptr ? cross_scale[l] : 1.f;
  if constexpr (KM == 32) {
    // one warp per row, lane s holding entry s: 32 values per thread do not fit in registers
    // next to the unrolled substitutions, so they move between lanes by shuffles instead
    __shared__ float Lp[KM][KM + 1];  // Lf with a padded row: column reads without bank conflicts
    for (int e = threadIdx.x; e < KM * KM; e += CS_THREADS) Lp[e / KM][e % KM] = Lf[e / KM][e % KM];
    __syncthreads();
    const int lane = threadIdx.x & 31;
    const bool on = lane < k;
    constexpr int RW = 4;  // rows per warp at a time: four independent shuffle chains
    for (int64_t i0 = int64_t(threadIdx.x >> 5) * RW; i0 < d; i0 += (CS_THREADS / 32) * RW) {
      float c[RW];
#pragma unroll
      for (int r = 0; r < RW; ++r) {
        const int64_t i = i0 + r;
        float v = 0.f;
        if (on && i < d)
          for (int z = 0; z < nsplit; ++z) v += CAl[z * zs + i * k + lane];
        c[r] = v * cs;
      }
      if (Bp != nullptr) {
        float bl[RW];
#pragma unroll
        for (int r = 0; r < RW; ++r) bl[r] = (on && i0 + r < d) ? Bp[(i0 + r) * k + lane] : 0.f;
#pragma unroll
        for (int t = 0; t < KM; ++t) {
          const float g = Gf[t][lane];
#pragma unroll
          for (int r = 0; r < RW; ++r) c[r] = fmaf(__shfl_sync(0xffffffffu, bl[r], t), g, c[r]);
        }
#pragma unroll
        for (int r = 0; r < RW; ++r)
          if (!on) c[r] = 0.f;
      }
      if (C_out != nullptr && j == 0 && on)
#pragma unroll
        for (int r = 0; r < RW; ++r)
          if (i0 + r < d && LOCA_CHECK((int64_t(l) * d + i0 + r) * k + lane, int64_t(L) * d * k))
            C_out[(int64_t(l) * d + i0 + r) * k + lane] = c[r];
      if (inf != 0) {
#pragma unroll
        for (int r = 0; r < RW; ++r)
          if (on && i0 + r < d) Bj[(i0 + r) * k + lane] = 0.f;
        continue;
      }
      // c <- c (L L^T)^-1: forward L y = c^T, then L^T x = y
#pragma unroll
      for (int t = 0; t < KM; ++t) {
        const float lt = Lp[lane][t], it = Linv[t];
#pragma unroll
        for (int r = 0; r < RW; ++r) {
          if (lane == t) c[r] *= it;
          const float yt = __shfl_sync(0xffffffffu, c[r], t);
          if (lane > t) c[r] = fmaf(-lt, yt, c[r]);
        }
      }
#pragma unroll
      for (int t = KM - 1; t >= 0; --t) {
        const float lt = Lp[t][lane], it = Linv[t];
#pragma unroll
        for (int r = 0; r < RW; ++r) {
          if (lane == t) c[r] *= it;
          const float xt = __shfl_sync(0xffffffffu, c[r], t);
          if (lane < t) c[r] = fmaf(-lt, xt, c[r]);
        }
      }
#pragma unroll
      for (int r = 0; r < RW; ++r)
        if (on && i0 + r < d && LOCA_CHECK((i0 + r) * k + lane, d * k)) Bj[(i0 + r) * k + lane] = c[r];
    }
  } else {
    for (int64_t i = threadIdx.x; i < d; i += CS_THREADS) {
      if (!LOCA_CHECK_SPAN(i * k, k, d * k) || !LOCA_CHECK_SPAN((int64_t(j) * L + l) * d * k + i * k, k,
                                                               int64_t(gridDim.x) * L * d * k))
        break;
      float c[KM];
#pragma unroll
      for (int s = 0; s < KM; ++s) c[s] = 0.f;
#pragma unroll 1
      for (int z = 0; z < nsplit; ++z) {
        const float* cz = CAl + z * zs + i * k;
#pragma unroll
        for (int s = 0; s < KM; ++s)
          if (s < k) c[s] += cz[s];
      }
#pragma unroll
      for (int s = 0; s < KM; ++s) c[s] *= cs;
      if (Bp != nullptr) {
        float b[KM];
#pragma unroll
        for (int s = 0; s < KM; ++s) b[s] = (s < k) ? Bp[i * k + s] : 0.f;
#pragma unroll
        for (int s = 0; s < KM; ++s) {
          float a = c[s];
#pragma unroll
          for (int t = 0; t < KM; ++t) a = fmaf(b[t], Gf[t][s], a);
          c[s] = (s < k) ? a : 0.f;
        }
      }
      if (C_out != nullptr && j == 0 && LOCA_CHECK_SPAN((int64_t(l) * d + i) * k, k, int64_t(L) * d * k)) {
#pragma unroll
        for (int s = 0; s < KM; ++s)
          if (s < k) C_out[(int64_t(l) * d + i) * k + s] = c[s];
      }
      if (inf != 0) {
#pragma unroll
        for (int s = 0; s < KM; ++s)
          if (s < k) Bj[i * k + s] = 0.f;
        continue;
      }
      chol_solve_row<KM>(Lf, Linv, c);
#pragma unroll
      for (int s = 0; s < KM; ++s)
        if (s < k) Bj[i * k + s] = c[s];
    }
  }
}

template <int KM>
cudaError_t project_t(const float* gram, const float* cross, const float* A, int L, int64_t d,
                      int k, float* GA, float* CA, cudaStream_t s) {
  const dim3 grid = dim3(unsigned((2 * d + PR_ROWS - 1) / PR_ROWS), unsigned(L), unsigned(PR_SPLIT));
  const size_t smem = sizeof(float) * (size_t(PR_ROWS) * PR_LD + size_t(PR_JC) * KM);
  cudaError_t e = cudaFuncSetAttribute(k_project_rows<KM>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  k_project_rows<KM><<<grid, PR_THREADS, smem, s>>>(gram, cross, A, d, k, GA, CA);
  return cudaGetLastError();
}

template <int KM>
cudaError_t solve_t(const float* GA, const float* CA, int nsplit, const float* A, const float* B_prev,
                    const double* xsq_total, const float* cross_scale, const float* lr, int nl, int L,
                    int64_t d, int k, float* B, int32_t* info, float* G_out, float* C_out, cudaStream_t s) {
  float v[16] = {};
  for (int i = 0; i < nl && i < 16; ++i) v[i] = lr[i];
  const dim3 grid = dim3(unsigned(nl), unsigned(L));
  k_chol_solve<KM><<<grid, CS_THREADS, 0, s>>>(GA, CA, nsplit, A, B_prev, xsq_total, cross_scale, d, k, L, v[0], v[1],
                                               v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9],
                                               v[10], v[11], v[12], v[13], v[14], v[15], B, info,
                                               G_out, C_out);
  return cudaGetLastError();
}

}  // namespace

int project_split() { return PR_SPLIT; }

cudaError_t launch_project_rows(const float* gram, const float* cross, const float* A, int L,
                                int64_t d, int k, float* GA, float* CA, cudaStream_t s) {
  if (k <= 4) return project_t<4>(gram, cross, A, L, d, k, GA, CA, s);
  if (k <= 8) return project_t<8>(gram, cross, A, L, d, k, GA, CA, s);
  if (k <= 16) return project_t<16>(gram, cross, A, L, d, k, GA, CA, s);
  if (k <= 32) return project_t<32>(gram, cross, A, L, d, k, GA, CA, s);
  return project_t<64>(gram, cross, A, L, d, k, GA, CA, s);
}

cudaError_t launch_chol_solve(const float* GA, const float* CA, int nsplit, const float* A, const float* B_prev,
                              const double* xsq_total, const float* cross_scale, const float* lambda_rel,
                              int nl, int L, int64_t d, int k, float* B, int32_t* info, float* G_out,
                              float* C_out, cudaStream_t s) {
#define LOCA_SOLVE(KM)                                                                               \
  return solve_t<KM>(GA, CA, nsplit, A, B_prev, xsq_total, cross_scale, lambda_rel, nl, L, d, k, B, info, G_out, \
                     C_out, s)
  if (k <= 4) LOCA_SOLVE(4);
  if (k <= 8) LOCA_SOLVE(8);
  if (k <= 16) LOCA_SOLVE(16);
  LOCA_SOLVE(32);
#undef LOCA_SOLVE
}

}  // namespace loca
