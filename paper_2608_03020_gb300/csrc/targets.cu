// Tokenwise feedback predictions of every block (S3: Q_l := F_l E), applied through the
// low-rank factors (S11: F e = U_k (S_k (V_k^T e))):  T_l = (E P_l) Q_l.
//
// k_qqt        M_l = Q_l Q_l^T (r x r), so that ||T_l||^2 = sum_n u_n^T M_l u_n with u_n = E[n] P_l.
// k_targets    persistent; a work item is (block l, 256-channel tile, 1024-token chunk).  The
//              tile Q_l[:, j0:j0+256] stays in shared memory for the item; for each 64-token
//              tile the E rows (prefetched into registers one tile ahead) give U = E P_l
//              (64 x r) in shared memory, and each thread forms an 8 token x 8 channel register
//              tile of T = U Q_l (fp32 FMA), rounds once to the output type and stores it (a
//              warp writes two runs of 256 contiguous bytes per token row in bf16).  Items of
//              channel tile 0 also
//              reduce u^T M_l u over their tokens into one partial; a second kernel sums the
//              partials in a fixed order (deterministic).
// Bound: 2 r fp32 FMA-flops per output element and 2 (bf16) or 4 (fp32) output bytes: at
// r = 16 with bf16 output the FMA pipe (~128 FMA/clk/SM) is the limit, not HBM.
#include <cuda_bf16.h>

#include "loca_internal.h"

namespace loca {
namespace {

constexpr int TN = 64;         // tokens per tile
constexpr int TD = 256;        // channels per tile
constexpr int CHUNK = 1024;    // tokens per work item
constexpr int kMaxC = 64;      // label columns supported by the fused U stage

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// M_l = Q_l Q_l^T, one thread block per block l.
__global__ void __launch_bounds__(256) k_qqt(const float* __restrict__ Q, int r, int64_t d,
                                             float* __restrict__ M) {
  const int l = blockIdx.x;
  const float* Ql = Q + int64_t(l) * r * d;
  for (int e = threadIdx.x; e < r * r; e += 256) {
    const int a = e / r, b = e % r;
    if (b < a) continue;
    const float* qa = Ql + int64_t(a) * d;
    const float* qb = Ql + int64_t(b) * d;
    double acc = 0.0;
    float part = 0.f;
    for (int64_t j = 0; j < d; ++j) {
      part = fmaf(qa[j], qb[j], part);
      if ((j & 63) == 63) { acc += part; part = 0.f; }
    }
    acc += part;
    M[(int64_t(l) * r + a) * r + b] = float(acc);
    M[(int64_t(l) * r + b) * r + a] = float(acc);
  }
}

template <bool kBF16>
__global__ void __launch_bounds__(256, 2) k_targets(const float* __restrict__ E, int64_t N, int C,
                                                    const float* __restrict__ P,
                                                    const float* __restrict__ Q,
                                                    const float* __restrict__ M, int r, int64_t d,
                                                    int L, void* __restrict__ Tout,
                                                    double* __restrict__ partials) {
  extern __shared__ float smem[];
  float* q_s = smem;                 // r x TD
  float* u_s = q_s + r * TD;         // r x TN (transposed U tile)
  float* e_s = u_s + TN * r;         // TN x C
  float* p_s = e_s + TN * kMaxC;     // C x r
  float* m_s = p_s + kMaxC * r;      // r x r
  __shared__ double red[8];
  const int t = threadIdx.x;
  const int cg = t & 31, tg = t >> 5;
  const int64_t nd = (d + TD - 1) / TD;
  const int64_t nchunks = (N + CHUNK - 1) / CHUNK;
  const int64_t items = int64_t(L) * nd * nchunks;

  for (int64_t it = blockIdx.x; it < items; it += gridDim.x) {
    const int l = int(it / (nd * nchunks));
    const int64_t rem = it - int64_t(l) * nd * nchunks;
    const int64_t jt = rem / nchunks;
    const int64_t ck = rem - jt * nchunks;
    const int64_t j0 = jt * TD;
    const int64_t nbeg = ck * CHUNK;
    const int64_t nend = (nbeg + CHUNK < N) ? nbeg + CHUNK : N;
    const bool do_sq = (jt == 0) && partials != nullptr;
    const float* Ql = Q + int64_t(l) * r * d;
    const float* Pl = P + int64_t(l) * C * r;

    __syncthreads();  // previous item's shared-memory readers are done
    for (int e = t; e < r * TD; e += 256) {
      const int s = e / TD, jj = e - s * TD;
      q_s[e] = (j0 + jj < d) ? Ql[int64_t(s) * d + j0 + jj] : 0.f;
    }
    for (int e = t; e < C * r; e += 256) p_s[e] = Pl[e];
    if (do_sq)
      for (int e = t; e < r * r; e += 256) m_s[e] = M[int64_t(l) * r * r + e];
    // E rows of the first tile
    float ev[(TN * kMaxC) / 256];
    const int nev = (TN * C + 255) / 256;
#pragma unroll
    for (int i = 0; i < (TN * kMaxC) / 256; ++i) {
      const int e = t + 256 * i;
      ev[i] = (i < nev && e < TN * C && nbeg + e / C < nend) ? E[nbeg * C + e] : 0.f;
    }
    float sq = 0.f;
    for (int64_t n0 = nbeg; n0 < nend; n0 += TN) {
      // stage E tile, then U = E P_l
#pragma unroll
      for (int i = 0; i < (TN * kMaxC) / 256; ++i) {
        const int e = t + 256 * i;
        if (i < nev && e < TN * C) e_s[e] = ev[i];
      }
      __syncthreads();
      for (int e = t; e < TN * r; e += 256) {
        const int s = e / TN, nn = e - s * TN;
        float u = 0.f;
        for (int c = 0; c < C; ++c) u = fmaf(e_s[nn * C + c], p_s[c * r + s], u);
        u_s[e] = u;  // transposed: u_s[s * TN + token]
      }
      // prefetch the next tile's E rows
      const int64_t n1 = n0 + TN;
#pragma unroll
      for (int i = 0; i < (TN * kMaxC) / 256; ++i) {
        const int e = t + 256 * i;
        ev[i] = (i < nev && e < TN * C && n1 + e / C < nend) ? E[n1 * C + e] : 0.f;
      }
      __syncthreads();
      if (do_sq && t < TN && n0 + t < nend) {
        // ||t_n||^2 = u_n^T M_l u_n for this thread's token
        float acc = 0.f;
        for (int a = 0; a < r; ++a) {
          float ma = 0.f;
          for (int b = 0; b < r; ++b) ma = fmaf(m_s[a * r + b], u_s[b * TN + t], ma);
          acc = fmaf(u_s[a * TN + t], ma, acc);
        }
        sq += acc;
      }
      // T tile: 8 tokens x 8 channels per thread
      float acc[8][8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int jj = 0; jj < 8; ++jj) acc[i][jj] = 0.f;
#pragma unroll 4
      for (int s = 0; s < r; ++s) {
        // this thread's 8 tokens: two broadcast 16-byte loads; its 8 channels: 4 at cg*4 and 4
        // at 128 + cg*4 (a warp reads 2 x 512 consecutive bytes: no bank conflicts)
        const float4 ua = *reinterpret_cast<const float4*>(u_s + s * TN + tg * 8);
        const float4 ub = *reinterpret_cast<const float4*>(u_s + s * TN + tg * 8 + 4);
        const float u[8] = {ua.x, ua.y, ua.z, ua.w, ub.x, ub.y, ub.z, ub.w};
        const float4 qa = *reinterpret_cast<const float4*>(q_s + s * TD + cg * 4);
        const float4 qb = *reinterpret_cast<const float4*>(q_s + s * TD + 128 + cg * 4);
        const float q[8] = {qa.x, qa.y, qa.z, qa.w, qb.x, qb.y, qb.z, qb.w};
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) acc[i][jj] = fmaf(u[i], q[jj], acc[i][jj]);
      }
      // channels jA = j0 + cg*4 .. +3 (acc[i][0..3]) and jB = j0 + 128 + cg*4 .. +3 (acc[i][4..7])
      const int64_t jA = j0 + cg * 4, jB = j0 + 128 + cg * 4;
      const bool fullA = (jA + 4 <= d) && (d % 4 == 0), fullB = (jB + 4 <= d) && (d % 4 == 0);
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int64_t n = n0 + tg * 8 + i;
        if (n >= nend) continue;
        const int64_t row = (int64_t(l) * N + n) * d;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          const int64_t jb = h ? jB : jA;
          const bool full = h ? fullB : fullA;
          const float* a = &acc[i][4 * h];
          if (full) {
            if (kBF16) {
              uint2 v;
              v.x = pack_bf16x2(a[0], a[1]);
              v.y = pack_bf16x2(a[2], a[3]);
              *reinterpret_cast<uint2*>(static_cast<__nv_bfloat16*>(Tout) + row + jb) = v;
            } else {
              *reinterpret_cast<float4*>(static_cast<float*>(Tout) + row + jb) = make_float4(a[0], a[1], a[2], a[3]);
            }
          } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              if (jb + u >= d) break;
              if (kBF16)
                static_cast<__nv_bfloat16*>(Tout)[row + jb + u] = __float2bfloat16_rn(a[u]);
              else
                static_cast<float*>(Tout)[row + jb + u] = a[u];
            }
          }
        }
      }
      __syncthreads();  // u_s and e_s are rewritten by the next tile
    }
    if (do_sq) {
      double dsq = sq;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) dsq += __shfl_xor_sync(0xffffffffu, dsq, off);
      if ((t & 31) == 0) red[t >> 5] = dsq;
      __syncthreads();
      if (t == 0) {
        double a = 0.0;
        for (int i = 0; i < 8; ++i) a += red[i];
        partials[int64_t(l) * nchunks + ck] = a;
      }
    }
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
  (void)d;
  return (N + CHUNK - 1) / CHUNK;
}

size_t targets_workspace_bytes(int64_t N, int L, int r) {
  return align256(sizeof(double) * size_t(L) * size_t(targets_num_partials(N, 0))) +
         align256(sizeof(float) * size_t(L) * size_t(r) * size_t(r));
}

int targets_max_C() { return kMaxC; }

cudaError_t launch_targets(const float* E, int64_t N, int C, const float* P, const float* Q,
                           int L, int r, int64_t d, void* T, int t_dtype, double* tsq,
                           void* workspace, cudaStream_t s) {
  if (N == 0 || d == 0) {
    if (tsq) return cudaMemsetAsync(tsq, 0, sizeof(double) * L, s);
    return cudaSuccess;
  }
  double* partials = nullptr;
  float* M = nullptr;
  cudaError_t e;
  if (tsq) {
    partials = static_cast<double*>(workspace);
    M = reinterpret_cast<float*>(static_cast<char*>(workspace) +
                                 align256(sizeof(double) * size_t(L) * size_t(targets_num_partials(N, d))));
    k_qqt<<<L, 256, 0, s>>>(Q, r, d, M);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  const int64_t items = int64_t(L) * ((d + TD - 1) / TD) * ((N + CHUNK - 1) / CHUNK);
  int64_t grid = int64_t(sm_count()) * 2;
  if (grid > items) grid = items;
  const size_t shm = sizeof(float) * size_t(r * TD + TN * r + TN * kMaxC + kMaxC * r + r * r);
  if (t_dtype == LOCA_BF16) {
    e = cudaFuncSetAttribute(k_targets<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets<true><<<unsigned(grid), 256, shm, s>>>(E, N, C, P, Q, M, r, d, L, T, partials);
  } else {
    e = cudaFuncSetAttribute(k_targets<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets<false><<<unsigned(grid), 256, shm, s>>>(E, N, C, P, Q, M, r, d, L, T, partials);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess || tsq == nullptr) return e;
  k_reduce_partials<<<L, 256, 0, s>>>(partials, targets_num_partials(N, d), tsq);
  return cudaGetLastError();
}

}  // namespace loca
