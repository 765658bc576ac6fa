// Projected statistics and batched positive-definite solves (Eqs. 8 and 9; Theorem S6; S7).
//
// k_project_rows  (shapes the tensor-core projection of project_tc.cu does not take: d or k not a
//                 multiple of 4, unaligned pointers)
//                 GA_l = Gram_l A_l, CA_l = Cross_l A_l (d x k each), as PR_SPLIT partial
//                 products over quarters of the column range (GA = sum_z GA_z, summed in a fixed
//                 order by k_chol_gram and k_chol_rows).  A CTA takes 256 rows of the stacked [Gram_l; Cross_l]
//                 and one column quarter; 32-column slabs of its rows are staged in shared memory
//                 by row-contiguous 16-byte loads (a warp request covers 4 rows, so L1 sees 4
//                 lines per request, not 32), then each thread forms a register block of
//                 RPT rows x SPT columns of the product with A's slab (broadcast reads).  Bound: the
//                 HBM read of Gram and Cross (8 d^2 bytes per block).
// k_chol_gram     G_l = A_l^T GA_l (k x k) as partial sums over chunks of the d rows: grid
//                 (chunks, L), GA_l summed over its nsplit partial products (fixed order) as the
//                 rows are staged; each chunk's k x k partial sum goes to the workspace.
// k_chol_factor   one thread block per (ridge candidate j, block l): the chunks' partial sums
//                 added in chunk order, lambda from the trace, Cholesky of G_l + lambda I in fp64
//                 in shared memory; the fp32 factor, its diagonal reciprocals and G_l go to a
//                 per-candidate record in the workspace.
// k_chol_rows     one thread per row i of C_l = B_prev,l G_l + s_l CA_l (s_l = cross_scale[l], or 1),
//                 solved by a forward and a back substitution against the staged factor:
//                 B[j, l, i] = C_l[i] (G_l + lambda I)^-1.  k is padded to a compile-time size with
//                 an identity block (its solution columns are zero), so each row stays in registers;
//                 d / 128 x nl x L thread blocks keep the SMs busy.
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

// Partial G_l = A_l^T GA_l over one chunk of rows: grid (nch, L); rows staged 128 at a time;
// a thread owns a 2 x 2 block of entries (KM = 32) or one entry (KM <= 16), fp32 over the chunk.
constexpr int GP_THREADS = 256;
constexpr int GP_ROWS = 128;
constexpr int GP_MAX_CHUNKS = 32;

template <int KM>
__global__ void __launch_bounds__(GP_THREADS) k_chol_gram(const float* __restrict__ GA, int nsplit,
                                                          const float* __restrict__ A, int64_t d, int k, int L,
                                                          float* __restrict__ gpart) {
  __shared__ __align__(16) float As[GP_ROWS][KM];
  __shared__ __align__(16) float Gs[GP_ROWS][KM];
  const int ch = blockIdx.x, l = blockIdx.y, nch = gridDim.x, tid = threadIdx.x;
  const int64_t per = (d + nch - 1) / nch;
  const int64_t r0 = int64_t(ch) * per, r1 = r0 + per < d ? r0 + per : d;
  const float* Al = A + int64_t(l) * d * k;
  const float* GAl = GA + int64_t(l) * d * k;
  const int64_t zs = int64_t(L) * d * k;  // stride between the nsplit partial products
  constexpr bool kBlk = KM == 32;
  const int a0 = kBlk ? (tid / 16) * 2 : tid / KM, b0 = kBlk ? (tid % 16) * 2 : tid % KM;
  const bool act = kBlk || tid < KM * KM;
  float g00 = 0.f, g01 = 0.f, g10 = 0.f, g11 = 0.f;
  for (int64_t i0 = r0; i0 < r1; i0 += GP_ROWS) {
    __syncthreads();
    for (int e = tid; e < GP_ROWS * KM; e += GP_THREADS) {
      const int ii = e / KM, s2 = e % KM;
      const bool ok = (i0 + ii < r1) && s2 < k && LOCA_CHECK((i0 + ii) * k + s2, d * k);
      As[ii][s2] = ok ? Al[(i0 + ii) * k + s2] : 0.f;
      float gsum = 0.f;
      if (ok)
        for (int z = 0; z < nsplit; ++z) gsum += GAl[z * zs + (i0 + ii) * k + s2];
      Gs[ii][s2] = gsum;
    }
    __syncthreads();
    if (act) {
      if constexpr (kBlk) {
#pragma unroll 8
        for (int ii = 0; ii < GP_ROWS; ++ii) {
          const float2 av = *reinterpret_cast<const float2*>(&As[ii][a0]);
          const float2 gv = *reinterpret_cast<const float2*>(&Gs[ii][b0]);
          g00 = fmaf(av.x, gv.x, g00);
          g01 = fmaf(av.x, gv.y, g01);
          g10 = fmaf(av.y, gv.x, g10);
          g11 = fmaf(av.y, gv.y, g11);
        }
      } else {
#pragma unroll 8
        for (int ii = 0; ii < GP_ROWS; ++ii) g00 = fmaf(As[ii][a0], Gs[ii][b0], g00);
      }
    }
  }
  float* out = gpart + (int64_t(l) * nch + ch) * KM * KM;
  if (kBlk) {
    out[a0 * KM + b0] = g00;
    out[a0 * KM + b0 + 1] = g01;
    out[(a0 + 1) * KM + b0] = g10;
    out[(a0 + 1) * KM + b0 + 1] = g11;
  } else if (act) {
    out[a0 * KM + b0] = g00;
  }
}

// Per-candidate factor record in the workspace: Lf (KM x KM fp32 lower factor), Linv (KM), and
// G_l (KM x KM fp32, symmetrised) for the B_prev term of the rows.
template <int KM>
__host__ __device__ constexpr int fac_floats() { return 2 * KM * KM + KM; }

template <int KM>
__global__ void __launch_bounds__(CS_THREADS) k_chol_factor(
    const float* __restrict__ gpart, int nch, const double* __restrict__ xsq_total,
    int64_t d, int k, int L,
    float l0, float l1, float l2, float l3, float l4, float l5, float l6, float l7, float l8,
    float l9, float l10, float l11, float l12, float l13, float l14, float l15,
    int32_t* __restrict__ info, float* __restrict__ G_out, float* __restrict__ fac) {
  __shared__ float Gf[KM][KM];   // G_l (fp32, symmetrised), padded with identity
  __shared__ double Md[KM][KM];  // G_l + lambda I, then its Cholesky factor (lower)
  __shared__ float Lf[KM][KM];
  __shared__ float Linv[KM];
  __shared__ int s_info;
  const int j = blockIdx.x, l = blockIdx.y;
  const float lam_rel[16] = {l0, l1, l2, l3, l4, l5, l6, l7, l8, l9, l10, l11, l12, l13, l14, l15};
  // G_l = A_l^T GA_l from the row chunks' partial products, summed in a fixed order in fp64
  const float* gp = gpart + int64_t(l) * nch * KM * KM;
  for (int e = threadIdx.x; e < KM * KM; e += CS_THREADS) {
    double acc = 0.0;
    for (int c = 0; c < nch; ++c) acc += double(gp[int64_t(c) * KM * KM + e]);
    Gf[e / KM][e % KM] = float(acc);
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

  float* f = fac + (int64_t(j) * L + l) * fac_floats<KM>();
  for (int e = threadIdx.x; e < KM * KM; e += CS_THREADS) {
    const int a = e / KM, b = e % KM;
    f[e] = Lf[a][b];
    f[KM * KM + KM + e] = (a < k && b < k) ? float(0.5 * (double(Gf[a][b]) + double(Gf[b][a]))) : 0.f;
  }
  for (int a = threadIdx.x; a < KM; a += CS_THREADS) f[KM * KM + a] = Linv[a];
}

// Rows of B for one (ridge candidate j, block l): thread per row i,
//   c = s_l CA_l[i] (+ B_prev,l[i] G_l),  B[j, l, i] = c (L L^T)^-1
// with the candidate's factor staged in shared memory (broadcast reads); C_out = c for j = 0.
constexpr int CR_THREADS = 128;

template <int KM>
__global__ void __launch_bounds__(CR_THREADS) k_chol_rows(
    const float* __restrict__ CA, int nsplit, const float* __restrict__ B_prev, const float* __restrict__ cross_scale,
    int64_t d, int k, int L, const int32_t* __restrict__ info, const float* __restrict__ fac, float* __restrict__ B,
    float* __restrict__ C_out) {
  __shared__ float Lf[KM][KM];
  __shared__ float Linv[KM];
  __shared__ float Gf[KM][KM];
  const int j = blockIdx.y, l = blockIdx.z;
  const float* f = fac + (int64_t(j) * L + l) * fac_floats<KM>();
  for (int e = threadIdx.x; e < KM * KM; e += CR_THREADS) {
    Lf[e / KM][e % KM] = f[e];
    Gf[e / KM][e % KM] = f[KM * KM + KM + e];
  }
  for (int a = threadIdx.x; a < KM; a += CR_THREADS) Linv[a] = f[KM * KM + a];
  __syncthreads();
  const int inf = info[int64_t(j) * L + l];
  const int64_t zs = int64_t(L) * d * k;  // stride between the nsplit partial products
  const float cs = cross_scale != nullptr ? cross_scale[l] : 1.f;
  float* Bj = B + (int64_t(j) * L + l) * d * k;
  const int64_t i = int64_t(blockIdx.x) * CR_THREADS + threadIdx.x;
  if (i >= d) return;
  if (!LOCA_CHECK_SPAN((int64_t(l) * d + i) * k, k, int64_t(L) * d * k) ||
      !LOCA_CHECK_SPAN((int64_t(j) * L + l) * d * k + i * k, k, int64_t(gridDim.y) * L * d * k))
    return;
  const float* cz = CA + (int64_t(l) * d + i) * k;
  float c[KM];
#pragma unroll
  for (int s2 = 0; s2 < KM; ++s2) c[s2] = 0.f;
  for (int z = 0; z < nsplit; ++z) {
#pragma unroll
    for (int s2 = 0; s2 < KM; ++s2)
      if (s2 < k) c[s2] += cz[z * zs + s2];
  }
#pragma unroll
  for (int s2 = 0; s2 < KM; ++s2) c[s2] *= cs;
  if (B_prev != nullptr) {
    // c += B_prev,l[i] G_l, one entry of the B_prev row at a time (only c stays in registers)
    const float* bp = B_prev + (int64_t(l) * d + i) * k;
#pragma unroll 4
    for (int t = 0; t < k; ++t) {
      const float bt = bp[t];
#pragma unroll
      for (int s2 = 0; s2 < KM; ++s2) c[s2] = fmaf(bt, Gf[t][s2], c[s2]);
    }
  }
  if (C_out != nullptr && j == 0) {
#pragma unroll
    for (int s2 = 0; s2 < KM; ++s2)
      if (s2 < k) C_out[(int64_t(l) * d + i) * k + s2] = c[s2];
  }
  float* bj = Bj + i * k;
  if (inf != 0) {
#pragma unroll
    for (int s2 = 0; s2 < KM; ++s2)
      if (s2 < k) bj[s2] = 0.f;
    return;
  }
  chol_solve_row<KM>(Lf, Linv, c);
#pragma unroll
  for (int s2 = 0; s2 < KM; ++s2)
    if (s2 < k) bj[s2] = c[s2];
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
                    int64_t d, int k, float* B, int32_t* info, float* G_out, float* C_out, float* fac,
                    cudaStream_t s) {
  float v[16] = {};
  for (int i = 0; i < nl && i < 16; ++i) v[i] = lr[i];
  float* gpart = fac + size_t(16) * size_t(L) * size_t(fac_floats<32>());
  int64_t nch = (int64_t(sm_count()) * 2 + L - 1) / L;  // two chunk CTAs per SM over the blocks
  const int64_t maxch = (d + GP_ROWS - 1) / GP_ROWS;
  if (nch > maxch) nch = maxch;
  if (nch > GP_MAX_CHUNKS) nch = GP_MAX_CHUNKS;
  if (nch < 1) nch = 1;
  k_chol_gram<KM><<<dim3(unsigned(nch), unsigned(L)), GP_THREADS, 0, s>>>(GA, nsplit, A, d, k, L, gpart);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_chol_factor<KM><<<dim3(unsigned(nl), unsigned(L)), CS_THREADS, 0, s>>>(
      gpart, int(nch), xsq_total, d, k, L, v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], v[10], v[11],
      v[12], v[13], v[14], v[15], info, G_out, fac);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int64_t rows_per_cta = CR_THREADS;
  const dim3 grid = dim3(unsigned((d + rows_per_cta - 1) / rows_per_cta), unsigned(nl), unsigned(L));
  k_chol_rows<KM><<<grid, CR_THREADS, 0, s>>>(CA, nsplit, B_prev, cross_scale, d, k, L, info, fac, B, C_out);
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

size_t chol_workspace_bytes(int L) {
  return sizeof(float) * size_t(L) * (size_t(16) * size_t(fac_floats<32>()) + size_t(GP_MAX_CHUNKS) * 32 * 32);
}

cudaError_t launch_chol_solve(const float* GA, const float* CA, int nsplit, const float* A, const float* B_prev,
                              const double* xsq_total, const float* cross_scale, const float* lambda_rel,
                              int nl, int L, int64_t d, int k, float* B, int32_t* info, float* G_out,
                              float* C_out, float* fac, cudaStream_t s) {
#define LOCA_SOLVE(KM)                                                                               \
  return solve_t<KM>(GA, CA, nsplit, A, B_prev, xsq_total, cross_scale, lambda_rel, nl, L, d, k, B, info, G_out, \
                     C_out, fac, s)
  if (k <= 4) LOCA_SOLVE(4);
  if (k <= 8) LOCA_SOLVE(8);
  if (k <= 16) LOCA_SOLVE(16);
  LOCA_SOLVE(32);
#undef LOCA_SOLVE
}

}  // namespace loca
