// Tokenwise feedback predictions of every block (S3: Q_l := F_l E), applied through the
// low-rank factors (S11: F e = U_k (S_k (V_k^T e))):  T_l = (E P_l) Q_l.
//
// Two-stage skinny product per thread block: a tile of 64 tokens x 256 channels of block l.
//   stage 1  U = E[tile] P_l        (64 x r, fp32, into shared memory)
//   stage 2  T = U Q_l[:, tile]     (64 x 256, fp32 register tile of 8 x 8 per thread)
// then one rounding to the output type and 16-byte stores (a warp writes 512 contiguous
// bytes of one token row).  ||T_l||^2 of the unrounded values is reduced per thread block
// into a partial and the partials are summed in a fixed order by a second kernel.
// Bound: 2 r fp32 FMA-flops and 2 (bf16) or 4 (fp32) output bytes per element; at r = 16
// with bf16 output the FMA pipe, not HBM, is the limit (16 flop/B > the FMA/HBM ridge).
#include <cuda_bf16.h>

#include "loca_internal.h"

namespace loca {
namespace {

constexpr int TN = 64;   // tokens per tile
constexpr int TD = 256;  // channels per tile

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

template <bool kBF16>
__global__ void __launch_bounds__(256) k_targets(const float* __restrict__ E, int64_t N, int C,
                                                 const float* __restrict__ P,
                                                 const float* __restrict__ Q, int r, int64_t d,
                                                 void* __restrict__ Tout,
                                                 double* __restrict__ partials) {
  extern __shared__ float smem[];
  float* u_s = smem;            // TN x r
  float* q_s = smem + TN * r;   // r x TD
  const int t = threadIdx.x;
  const int l = blockIdx.z;
  const int64_t n0 = int64_t(blockIdx.x) * TN;
  const int64_t j0 = int64_t(blockIdx.y) * TD;
  const float* Pl = P + int64_t(l) * C * r;
  const float* Ql = Q + int64_t(l) * r * d;

  // stage 1: U = E[n0:n0+TN] P_l
  for (int e = t; e < TN * r; e += 256) {
    const int nn = e / r, s = e - nn * r;
    float u = 0.f;
    if (n0 + nn < N) {
      const float* er = E + (n0 + nn) * C;
      for (int c = 0; c < C; ++c) u = fmaf(er[c], Pl[c * r + s], u);
    }
    u_s[e] = u;
  }
  // Q_l[:, j0:j0+TD]
  for (int e = t; e < r * TD; e += 256) {
    const int s = e / TD, jj = e - s * TD;
    q_s[e] = (j0 + jj < d) ? Ql[int64_t(s) * d + j0 + jj] : 0.f;
  }
  __syncthreads();

  // stage 2: 8 tokens x 8 channels per thread
  const int cg = t & 31, tg = t >> 5;
  float acc[8][8];
#pragma unroll
  for (int i = 0; i < 8; ++i)
#pragma unroll
    for (int jj = 0; jj < 8; ++jj) acc[i][jj] = 0.f;
  for (int s = 0; s < r; ++s) {
    float u[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) u[i] = u_s[(tg * 8 + i) * r + s];
    const float4 qa = *reinterpret_cast<const float4*>(q_s + s * TD + cg * 8);
    const float4 qb = *reinterpret_cast<const float4*>(q_s + s * TD + cg * 8 + 4);
    const float q[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) acc[i][jj] = fmaf(u[i], q[jj], acc[i][jj]);
  }

  // stores and the sum of squares of the unrounded values
  const int64_t jb = j0 + cg * 8;
  const bool full8 = (jb + 8 <= d) && (d % 8 == 0);
  float sq = 0.f;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int64_t n = n0 + tg * 8 + i;
    if (n >= N) continue;
    const int64_t base = (int64_t(l) * N + n) * d + jb;
    if (full8) {
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) sq = fmaf(acc[i][jj], acc[i][jj], sq);
      if (kBF16) {
        uint4 v;
        v.x = pack_bf16x2(acc[i][0], acc[i][1]);
        v.y = pack_bf16x2(acc[i][2], acc[i][3]);
        v.z = pack_bf16x2(acc[i][4], acc[i][5]);
        v.w = pack_bf16x2(acc[i][6], acc[i][7]);
        *reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(Tout) + base) = v;
      } else {
        float* o = static_cast<float*>(Tout) + base;
        *reinterpret_cast<float4*>(o) = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        *reinterpret_cast<float4*>(o + 4) = make_float4(acc[i][4], acc[i][5], acc[i][6], acc[i][7]);
      }
    } else {
#pragma unroll
      for (int jj = 0; jj < 8; ++jj) {
        if (jb + jj >= d) break;
        sq = fmaf(acc[i][jj], acc[i][jj], sq);
        if (kBF16)
          static_cast<__nv_bfloat16*>(Tout)[base + jj] = __float2bfloat16_rn(acc[i][jj]);
        else
          static_cast<float*>(Tout)[base + jj] = acc[i][jj];
      }
    }
  }
  if (partials == nullptr) return;
  double dsq = sq;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) dsq += __shfl_xor_sync(0xffffffffu, dsq, off);
  __shared__ double red[8];
  __syncthreads();
  if ((t & 31) == 0) red[t >> 5] = dsq;
  __syncthreads();
  if (t == 0) {
    double a = 0.0;
    for (int i = 0; i < 8; ++i) a += red[i];
    const int64_t nparts = int64_t(gridDim.x) * gridDim.y;
    partials[int64_t(l) * nparts + int64_t(blockIdx.x) * gridDim.y + blockIdx.y] = a;
  }
}

// out[l] = sum of partials[l * nparts : (l + 1) * nparts] in a fixed order.
__global__ void __launch_bounds__(256) k_reduce_partials(const double* __restrict__ partials,
                                                         int64_t nparts, double* __restrict__ out) {
  __shared__ double red[256];
  const int l = blockIdx.x;
  double a = 0.0;
  for (int64_t i = threadIdx.x; i < nparts; i += 256) a += partials[int64_t(l) * nparts + i];
  red[threadIdx.x] = a;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) red[threadIdx.x] += red[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) out[l] = red[0];
}

}  // namespace

int64_t targets_num_partials(int64_t N, int64_t d) {
  return ((N + TN - 1) / TN) * ((d + TD - 1) / TD);
}

cudaError_t launch_targets(const float* E, int64_t N, int C, const float* P, const float* Q,
                           int L, int r, int64_t d, void* T, int t_dtype, double* tsq,
                           double* partials, cudaStream_t s) {
  if (N == 0 || d == 0) {
    if (tsq) return cudaMemsetAsync(tsq, 0, sizeof(double) * L, s);
    return cudaSuccess;
  }
  const dim3 grid = dim3(unsigned((N + TN - 1) / TN), unsigned((d + TD - 1) / TD), unsigned(L));
  const size_t shm = sizeof(float) * size_t(TN * r + r * TD);
  double* part = tsq ? partials : nullptr;
  cudaError_t e;
  if (t_dtype == LOCA_BF16) {
    e = cudaFuncSetAttribute(k_targets<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets<true><<<grid, 256, shm, s>>>(E, N, C, P, Q, r, d, T, part);
  } else {
    e = cudaFuncSetAttribute(k_targets<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets<false><<<grid, 256, shm, s>>>(E, N, C, P, Q, r, d, T, part);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess || tsq == nullptr) return e;
  k_reduce_partials<<<L, 256, 0, s>>>(partials, targets_num_partials(N, d), tsq);
  return cudaGetLastError();
}

}  // namespace loca
