// In-probe alignment diagnostic (supplement, one-shot calibration of the feedback map): per block,
//   alpha_l = <G_l, T_l>_F / (||G_l||_F ||T_l||_F),   T_l = E P_l Q_l  (the feedback predictions),
// with G_l the exact hidden-state gradients at the probe positions.  T is formed element by
// element in registers (r FMAs each) and never written.
//
// k_align_part   grid (token chunk, 256-channel tile, block): each thread owns one channel of the
//                tile; per 32-token sub-chunk the CTA forms U = E P_l for those tokens in shared
//                memory, then every thread walks the tokens: t = U[n] . Q_l[:, j], g = G[n][j],
//                and sums g t, g g, t t (fp32 over the chunk; fp64 block reduction in a fixed
//                order), one partial triple per CTA.
// k_align_final  per block, the partial triples in a fixed order -> alpha_l (0 if a norm is 0).
// k_align_u      for error spaces wider than kMaxM (the paper's d-wide e): U_l = E P_l (Np x r per
//                block, fp32) first, tiled over 64 tokens x 64 error channels in shared memory;
//                k_align_part then reads U_l instead of forming E P_l itself.
#include "loca_internal.h"

namespace loca {
namespace {

constexpr int AL_THREADS = 256;  // channels per tile
constexpr int AL_SUB = 32;       // tokens staged at a time
constexpr int AL_CHUNK = 1024;   // tokens per CTA
constexpr int kMaxM = 64;      // error width formed in k_align_part itself
constexpr int kMaxWideM = 16384;
constexpr int kMaxR = 32;
constexpr int AU_TOK = 64;     // tokens per CTA of k_align_u
constexpr int AU_CH = 64;      // error channels staged per step

// U[l][n][s] = sum_c E[n][c] P_l[c][s] (fp32), U laid out L x Np x r.
template <int RP>
__global__ void __launch_bounds__(AL_THREADS) k_align_u(const float* __restrict__ E, const float* __restrict__ P,
                                                      int64_t Np, int m, int r, float* __restrict__ U) {
  __shared__ float Es[AU_TOK][AU_CH + 1];
  __shared__ float Ps[AU_CH][RP];
  constexpr int SG = AL_THREADS / AU_TOK;  // column groups
  constexpr int SPT = RP / SG;             // product columns per thread (RP >= 8)
  const int l = blockIdx.y, tid = threadIdx.x;
  const int tt = tid % AU_TOK, sg = tid / AU_TOK;
  const int64_t n0 = int64_t(blockIdx.x) * AU_TOK;
  const float* Pl = P + int64_t(l) * m * r;
  float acc[SPT];
#pragma unroll
  for (int i = 0; i < SPT; ++i) acc[i] = 0.f;
  for (int c0 = 0; c0 < m; c0 += AU_CH) {
    __syncthreads();
    for (int e = tid; e < AU_TOK * AU_CH; e += AL_THREADS) {
      const int t = e / AU_CH, c = e % AU_CH;
      Es[t][c] = (n0 + t < Np && c0 + c < m) ? E[(n0 + t) * m + c0 + c] : 0.f;
    }
    for (int e = tid; e < AU_CH * RP; e += AL_THREADS) {
      const int c = e / RP, s = e % RP;
      Ps[c][s] = (c0 + c < m && s < r) ? Pl[int64_t(c0 + c) * r + s] : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int c = 0; c < AU_CH; ++c) {
      const float ev = Es[tt][c];
#pragma unroll
      for (int i = 0; i < SPT; ++i) acc[i] = fmaf(ev, Ps[c][sg + SG * i], acc[i]);
    }
  }
  const int64_t n = n0 + tt;
  if (n >= Np) return;
#pragma unroll
  for (int i = 0; i < SPT; ++i) {
    const int s = sg + SG * i;
    if (s < r && LOCA_CHECK((int64_t(l) * Np + n) * r + s, int64_t(gridDim.y) * Np * r)) U[(int64_t(l) * Np + n) * r + s] = acc[i];
  }
}

// kU: E holds U (L x Np x r) and P is not used: the predictions' r-dimensional codes are read,
// not formed.
template <int RP, bool kU>
__global__ void __launch_bounds__(AL_THREADS) k_align_part(const float* __restrict__ E, const float* __restrict__ P,
                                                         const float* __restrict__ Q, const float* __restrict__ G,
                                                         int64_t Np, int m, int64_t d, int r, int nch, int ntile,
                                                         double* __restrict__ part) {
  __shared__ float Qs[RP][AL_THREADS];
  __shared__ float Ps[kMaxM][RP];
  __shared__ float Us[AL_SUB][RP];
  __shared__ double red[3][AL_THREADS / 32];
  const int ch = blockIdx.x, tile = blockIdx.y, l = blockIdx.z, tid = threadIdx.x;
  const int64_t j = int64_t(tile) * AL_THREADS + tid;
  const bool jv = j < d;
  for (int s = 0; s < RP; ++s) Qs[s][tid] = (s < r && jv) ? Q[(int64_t(l) * r + s) * d + j] : 0.f;
  if (!kU)
    for (int e = tid; e < kMaxM * RP; e += AL_THREADS) {
      const int c = e / RP, s = e % RP;
      Ps[c][s] = (c < m && s < r) ? P[(int64_t(l) * m + c) * r + s] : 0.f;
    }
  const int64_t n0 = int64_t(ch) * AL_CHUNK;
  const int64_t n1 = (n0 + AL_CHUNK < Np) ? n0 + AL_CHUNK : Np;
  const float* Gl = G + int64_t(l) * Np * d;
  float gt = 0.f, gg = 0.f, tt = 0.f;
  for (int64_t s0 = n0; s0 < n1; s0 += AL_SUB) {
    __syncthreads();
    for (int e = tid; e < AL_SUB * RP; e += AL_THREADS) {
      const int t = e / RP, s = e % RP;
      float acc = 0.f;
      if (kU) {
        if (s0 + t < n1 && s < r) acc = E[(int64_t(l) * Np + s0 + t) * r + s];
      } else if (s0 + t < n1) {
        for (int c = 0; c < m; ++c) acc = fmaf(E[(s0 + t) * m + c], Ps[c][s], acc);
      }
      Us[t][s] = acc;
    }
    __syncthreads();
    const int nt = int((n1 - s0) < AL_SUB ? (n1 - s0) : AL_SUB);
    for (int t = 0; t < nt; ++t) {
      float tv = 0.f;
#pragma unroll
      for (int s = 0; s < RP; ++s) tv = fmaf(Us[t][s], Qs[s][tid], tv);
      const float g = (jv && LOCA_CHECK((s0 + t) * d + j, Np * d)) ? Gl[(s0 + t) * d + j] : 0.f;
      gt = fmaf(g, tv, gt);
      gg = fmaf(g, g, gg);
      tt = fmaf(tv, tv, tt);
    }
  }
  double v[3] = {double(gt), double(gg), double(tt)};
#pragma unroll
  for (int q = 0; q < 3; ++q)
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v[q] += __shfl_xor_sync(0xffffffffu, v[q], off);
  if ((tid & 31) == 0)
    for (int q = 0; q < 3; ++q) red[q][tid >> 5] = v[q];
  __syncthreads();
  if (tid < 3) {
    double a = 0.0;
    for (int w = 0; w < AL_THREADS / 32; ++w) a += red[tid][w];
    if (LOCA_CHECK(((int64_t(l) * ntile + tile) * nch + ch) * 3 + tid, int64_t(gridDim.z) * ntile * nch * 3))
      part[((int64_t(l) * ntile + tile) * nch + ch) * 3 + tid] = a;
  }
}

__global__ void k_align_final(const double* __restrict__ part, int nparts, double* __restrict__ alpha) {
  const int l = blockIdx.x;
  if (threadIdx.x != 0) return;
  double gt = 0.0, gg = 0.0, tt = 0.0;
  for (int i = 0; i < nparts; ++i) {
    const double* p = part + (int64_t(l) * nparts + i) * 3;
    gt += p[0];
    gg += p[1];
    tt += p[2];
  }
  if (LOCA_CHECK(l, gridDim.x)) alpha[l] = (gg > 0.0 && tt > 0.0) ? gt / sqrt(gg * tt) : 0.0;
}

}  // namespace

int align_max_m() { return kMaxWideM; }
int align_max_r() { return kMaxR; }

static size_t part_bytes(int64_t Np, int64_t d, int L) {
  const int64_t nch = (Np + AL_CHUNK - 1) / AL_CHUNK;
  const int64_t ntile = (d + AL_THREADS - 1) / AL_THREADS;
  return align256(sizeof(double) * 3 * size_t(L) * size_t(nch) * size_t(ntile));
}

size_t align_workspace_bytes(int64_t Np, int m, int64_t d, int L, int r) {
  const size_t u = m > kMaxM ? align256(sizeof(float) * size_t(L) * size_t(Np) * size_t(r)) : 0;
  return part_bytes(Np, d, L) + u;
}

template <int RP>
static cudaError_t align_t(const float* E, const float* G, int64_t Np, int m, int64_t d, int L, const float* P,
                           const float* Q, int r, double* alpha, void* workspace, cudaStream_t s) {
  const int nch = int((Np + AL_CHUNK - 1) / AL_CHUNK);
  const int ntile = int((d + AL_THREADS - 1) / AL_THREADS);
  double* part = static_cast<double*>(workspace);
  const dim3 grid = dim3(unsigned(nch), unsigned(ntile), unsigned(L));
  if (m > kMaxM) {
    float* U = reinterpret_cast<float*>(static_cast<char*>(workspace) + part_bytes(Np, d, L));
    k_align_u<RP><<<dim3(unsigned((Np + AU_TOK - 1) / AU_TOK), unsigned(L)), AL_THREADS, 0, s>>>(E, P, Np, m, r, U);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_align_part<RP, true><<<grid, AL_THREADS, 0, s>>>(U, P, Q, G, Np, r, d, r, nch, ntile, part);
  } else {
    k_align_part<RP, false><<<grid, AL_THREADS, 0, s>>>(E, P, Q, G, Np, m, d, r, nch, ntile, part);
  }
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_align_final<<<L, 32, 0, s>>>(part, nch * ntile, alpha);
  return cudaGetLastError();
}

cudaError_t launch_alignment(const float* E, const float* G, int64_t Np, int m, int64_t d, int L, const float* P,
                             const float* Q, int r, double* alpha, void* workspace, cudaStream_t s) {
  if (Np == 0) return cudaMemsetAsync(alpha, 0, sizeof(double) * L, s);
  if (r <= 8) return align_t<8>(E, G, Np, m, d, L, P, Q, r, alpha, workspace, s);
  if (r <= 16) return align_t<16>(E, G, Np, m, d, L, P, Q, r, alpha, workspace, s);
  return align_t<32>(E, G, Np, m, d, L, P, Q, r, alpha, workspace, s);
}

}  // namespace loca
