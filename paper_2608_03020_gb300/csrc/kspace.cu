// The paper's own k-space statistics (Eqs. 6, 8, 9; S7, S8): per block l and mini-batch,
//
//   p_n   = A_l^T x_n                 (k)         Xp = X_l A_l   (N x k)
//   G_l  += sum_n p_n p_n^T           (k x k)     = Xp^T Xp
//   S_l  += alpha_l sum_n e_n p_n^T   (C x k)     = alpha_l E^T Xp,  alpha_l = -eta RMS(X_l)/RMS(T_l)
//   xsq_l += ||X_l||_F^2
//
// and the solve of B_l (G_l + lambda I) = C_l with C_l = B_prev,l G_l + Q_l^T (P_l^T S_l), which
// equals sum_n rho_n p_n^T with rho_n = B_prev p_n - eta_bar q_n and q_n = T_l[n] = (e_n P_l) Q_l
// (targets applied through the factors, S11).  T is never formed: ||T_l||^2 comes in closed form
// as sum_n u_n^T (Q_l Q_l^T) u_n with u_n = e_n P_l.  One HBM read of X per block is the work.
//
// Kernels:
//   k_kspace_prep   per block: W_l = A_l^T split into bf16 hi / lo rows (2 kp x d, kp = 16 or
//                   32; A_l ~= hi + lo to 2^-16), and M_l = Q_l Q_l^T (r x r), 8 CTAs per block.
//   k_kspace_xa     Xp = X_l W_l^T on tcgen05 (kind::f16, M = 128 tokens, N = 2 kp, K = 16, both
//                   operands K-major with the 128-byte swizzle): a persistent CTA per SM streams
//                   128-token x 64-channel tiles of X (16 KB) and the matching W tile through an
//                   8-stage TMA ring; the epilogue warps also sum the squares of every X tile
//                   from shared memory, and write p = hi-part + lo-part (fp32) per token.
//   k_kspace_stats  token-parallel partials of Xp^T Xp, E^T Xp and sum u^T M u (fp32 over 128
//                   tokens, fp64 across).
//   k_kspace_final  fixed-order reduction of all partials per block (deterministic), alpha_l,
//                   and the update of G, S, xsq_total.
//   k_kspace_solve  lambda from the trace, Cholesky of G_l + lambda I, C_l rows from Q_l^T (P_l^T
//                   S_l) (+ B_prev,l G_l), forward and back substitution per row.
// Every mbarrier wait is bounded (see tc_ptx.cuh).
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstring>

#include "chol.cuh"
#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

using namespace tc;

// ------------------------------------------------------------------ prep
constexpr int PREP_THREADS = 256;
constexpr int PREP_SPLIT = 8;  // CTAs per block

// grid (L, PREP_SPLIT): each CTA splits a slice of A_l^T and forms a slice of the r x r entries
// of Q_l Q_l^T, one warp per entry (lanes over channels; fp32 lane sums, fp64 across lanes).
__global__ void __launch_bounds__(PREP_THREADS) k_kspace_prep(const float* __restrict__ A, const float* __restrict__ Q,
                                                             int64_t d, int k, int kp, int r,
                                                             __nv_bfloat16* __restrict__ W, float* __restrict__ M) {
  const int l = blockIdx.x, part = blockIdx.y;
  const float* Al = A + int64_t(l) * d * k;
  __nv_bfloat16* Wl = W + int64_t(l) * 2 * kp * d;
  const int64_t tot = int64_t(kp) * d;
  for (int64_t e = int64_t(part) * PREP_THREADS + threadIdx.x; e < tot; e += int64_t(PREP_SPLIT) * PREP_THREADS) {
    const int s = int(e / d);
    const int64_t j = e - int64_t(s) * d;
    const float a = (s < k) ? Al[j * k + s] : 0.f;
    const __nv_bfloat16 hi = __float2bfloat16_rn(a);
    const __nv_bfloat16 lo = __float2bfloat16_rn(a - __bfloat162float(hi));
    Wl[int64_t(s) * d + j] = hi;
    Wl[int64_t(kp + s) * d + j] = lo;
  }
  const float* Ql = Q + int64_t(l) * r * d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int kWarps = PREP_THREADS / 32;
  for (int e = part * kWarps + warp; e < r * r; e += PREP_SPLIT * kWarps) {
    const int a = e / r, b = e % r;
    float acc = 0.f;
    for (int64_t j = lane; j < d; j += 32) acc = fmaf(Ql[int64_t(a) * d + j], Ql[int64_t(b) * d + j], acc);
    double v = double(acc);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    if (lane == 0) M[(int64_t(l) * r + a) * r + b] = float(v);
  }
}

// ------------------------------------------------------------------ X A on the tensor cores
constexpr int XA_THREADS = 192;
constexpr int XA_TM = 128;          // tokens per tile (TMEM lanes)
constexpr int XA_BK = 64;           // channels per stage (one 128-byte swizzle row)
constexpr int XA_STAGES = 8;
constexpr int XA_XBYTES = XA_TM * XA_BK * 2;  // 16 KB
constexpr int XA_STAGE = 24 * 1024;           // X tile + up to 64 W rows (8 KB)
constexpr int XA_SMEM = XA_STAGES * XA_STAGE + 1024 + 256;
constexpr uint32_t XA_TMEM_COLS = 128;

template <int KP>
__global__ void __launch_bounds__(XA_THREADS, 1)
    k_kspace_xa(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW, int L,
                int64_t N, int64_t d, int ntiles, float* __restrict__ Xp, double* __restrict__ xsq_part,
                int32_t* status, int32_t* abort_flag, unsigned long long limit_ns) {
  constexpr int NCOL = 2 * KP;
  constexpr uint32_t WBYTES = uint32_t(NCOL) * 128u;
  constexpr uint32_t ID = tc::idesc(1, 1, 0, 0, XA_TM, NCOL);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + XA_STAGES * XA_STAGE);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * XA_STAGES + 6);
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = smem_u32(bars);
  auto full_bar = [&](int s) { return bar0 + 8u * s; };
  auto empty_bar = [&](int s) { return bar0 + 8u * (XA_STAGES + s); };
  auto acc_full = [&](int b) { return bar0 + 8u * (2 * XA_STAGES + b); };
  auto acc_empty = [&](int b) { return bar0 + 8u * (2 * XA_STAGES + 2 + b); };
  const uint32_t drain_bar = bar0 + 8u * (2 * XA_STAGES + 4);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{status, abort_flag, limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < XA_STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 5);  // the MMA commit and lane 0 of the four epilogue warps
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), 4);
    }
    mbar_init(drain_bar, 1);
    mbar_init_fence();
    prefetch_tensormap(&tmX);
    prefetch_tensormap(&tmW);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), XA_TMEM_COLS);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int nkc = int((d + XA_BK - 1) / XA_BK);
  const int total = L * ntiles;

  if (warp == 0) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, pending = 0, pending_par = 0;
      bool ok = true;
      for (int it = blockIdx.x; it < total && ok; it += gridDim.x) {
        const int l = it / ntiles;
        const int t0 = (it - l * ntiles) * XA_TM;
        for (int kc = 0; kc < nkc; ++kc) {
          if (!mbar_try_wait(empty_bar(stage), phase ^ 1u) && !mbar_wait(empty_bar(stage), phase ^ 1u, wc)) {
            ok = false;
            break;
          }
          const uint32_t fb = full_bar(stage);
          mbar_arrive_expect_tx(fb, XA_XBYTES + WBYTES);
          pending |= 1u << stage;
          pending_par = (pending_par & ~(1u << stage)) | (phase << stage);
          const uint32_t st = sbase + uint32_t(stage) * XA_STAGE;
          tma_load_3d(st, &tmX, fb, kc * XA_BK, t0, l);
          tma_load_3d(st + XA_XBYTES, &tmW, fb, kc * XA_BK, 0, l);
          if (++stage == XA_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        for (int s = 0; s < XA_STAGES; ++s)
          if (pending & (1u << s)) mbar_drain(full_bar(s), (pending_par >> s) & 1u, limit_ns);
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, tcount = 0;
      bool ok = true, issued = false;
      for (int it = blockIdx.x; it < total && ok; it += gridDim.x, ++tcount) {
        const int buf = int(tcount & 1u);
        const uint32_t aph = (tcount >> 1) & 1u;
        if (!mbar_wait(acc_empty(buf), aph ^ 1u, wc)) { ok = false; break; }
        fence_after();
        const uint32_t dt = tmem_base + uint32_t(buf * NCOL);
        for (int kc = 0; kc < nkc; ++kc) {
          if (!mbar_try_wait(full_bar(stage), phase) && !mbar_wait(full_bar(stage), phase, wc)) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t st = sbase + uint32_t(stage) * XA_STAGE;
          const uint64_t a0 = sdesc(st, 16u, 1024u, kSwizzle128B);
          const uint64_t b0 = sdesc(st + XA_XBYTES, 16u, 1024u, kSwizzle128B);
#pragma unroll
          for (int kk = 0; kk < XA_BK / 16; ++kk)  // K = 16 slices advance 32 bytes within the row
            mma_f16(dt, a0 + uint64_t(kk * 2), b0 + uint64_t(kk * 2), ID, (kc | kk) != 0 ? 1u : 0u);
          issued = true;
          mma_commit(empty_bar(stage));
          if (++stage == XA_STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        mma_commit(acc_full(buf));
      }
      if (!ok && issued) {
        mma_commit(drain_bar);
        mbar_drain(drain_bar, 0, limit_ns);
      }
    }
    __syncwarp();
  } else {
    // epilogue warps 2..5: TMEM lane quarter q; token row = q * 32 + lane of each tile
    const int q = warp & 3;
    const int row = q * 32 + lane;
    int stage = 0;
    uint32_t phase = 0, tcount = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x, ++tcount) {
      const int l = it / ntiles;
      const int tile = it - l * ntiles;
      const int t0 = tile * XA_TM;
      double xs = 0.0;
      bool ok = true;
      for (int kc = 0; kc < nkc; ++kc) {
        const bool w_ok = mbar_wait(full_bar(stage), phase, wc);
        if (!__all_sync(0xffffffffu, w_ok)) { ok = false; break; }
        // squares of this token's 64 channels: row `row` of the swizzled tile (chunk order is
        // irrelevant for a sum, so lane i starts at chunk i % 8 and the 32 lanes' 16-byte reads
        // spread over all banks); zero-filled out-of-range tokens and channels add nothing
        const uint32_t ra = sbase + uint32_t(stage) * XA_STAGE + uint32_t(row >> 3) * 1024u + uint32_t(row & 7) * 128u;
        float part = 0.f;
#pragma unroll
        for (int c = 0; c < 8; ++c) {
          uint32_t w0, w1, w2, w3;
          asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(w0), "=r"(w1), "=r"(w2), "=r"(w3)
                       : "r"(ra + uint32_t((c + row) & 7) * 16u));
          const uint32_t wv[4] = {w0, w1, w2, w3};
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const float lo = __uint_as_float(wv[u] << 16), hi = __uint_as_float(wv[u] & 0xffff0000u);
            part = fmaf(lo, lo, part);
            part = fmaf(hi, hi, part);
          }
        }
        xs += double(part);
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar(stage));
        if (++stage == XA_STAGES) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      const int buf = int(tcount & 1u);
      const bool a_ok = mbar_wait(acc_full(buf), (tcount >> 1) & 1u, wc);
      if (!__all_sync(0xffffffffu, a_ok)) break;
      fence_after();
      float v[NCOL];
      const uint32_t ta = tmem_base + (uint32_t(q * 32) << 16) + uint32_t(buf * NCOL);
      if constexpr (NCOL == 32) {
        tmem_ld32(ta, v);
      } else {
        tmem_ld32x2(ta, v);
      }
      fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(acc_empty(buf));
      const int64_t n = int64_t(t0) + row;
      if (n < N) {
        float4* o = reinterpret_cast<float4*>(Xp + (int64_t(l) * N + n) * KP);
#pragma unroll
        for (int u = 0; u < KP / 4; ++u)
          o[u] = make_float4(v[4 * u] + v[KP + 4 * u], v[4 * u + 1] + v[KP + 4 * u + 1],
                             v[4 * u + 2] + v[KP + 4 * u + 2], v[4 * u + 3] + v[KP + 4 * u + 3]);
      }
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) xs += __shfl_xor_sync(0xffffffffu, xs, off);
      if (lane == 0) xsq_part[(int64_t(l) * ntiles + tile) * 4 + q] = xs;
    }
  }

  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, XA_TMEM_COLS);
}

// ------------------------------------------------------------------ token-parallel partials
constexpr int ST_THREADS = 256;
constexpr int ST_SUB = 128;    // tokens staged in shared memory at a time
constexpr int ST_CHUNK = 4096; // tokens per CTA
constexpr int kMaxCk = 16;     // C limit of the k-space path
constexpr int kMaxRk = 32;     // r limit

__host__ __device__ constexpr int part_stride(int kp, int C) { return kp * kp + C * kp + 1; }

template <int KP>
__global__ void __launch_bounds__(ST_THREADS) k_kspace_stats(const float* __restrict__ Xp, const float* __restrict__ E,
                                                           const float* __restrict__ P, const float* __restrict__ M,
                                                           int64_t N, int C, int r, int nch,
                                                           double* __restrict__ part) {
  __shared__ float xs[ST_SUB][KP + 1];
  __shared__ float es[ST_SUB][kMaxCk + 1];
  __shared__ float Ms[kMaxRk][kMaxRk + 1];
  __shared__ float Ps[kMaxCk][kMaxRk];
  __shared__ double red[ST_THREADS];
  const int ch = blockIdx.x, l = blockIdx.y;
  const int tid = threadIdx.x;
  for (int e = tid; e < r * r; e += ST_THREADS) Ms[e / r][e % r] = M[int64_t(l) * r * r + e];
  for (int e = tid; e < C * r; e += ST_THREADS) Ps[e / r][e % r] = P[int64_t(l) * C * r + e];
  constexpr int GPT = (KP * KP + ST_THREADS - 1) / ST_THREADS;
  const int SPT = (C * KP + ST_THREADS - 1) / ST_THREADS;  // <= 2 (C <= 16, KP <= 32)
  double g[GPT], sacc[2];
#pragma unroll
  for (int i = 0; i < GPT; ++i) g[i] = 0.0;
  sacc[0] = sacc[1] = 0.0;
  double tq = 0.0;
  const int64_t n_beg = int64_t(ch) * ST_CHUNK;
  const int64_t n_end = (n_beg + ST_CHUNK < N) ? n_beg + ST_CHUNK : N;
  const float* Xl = Xp + int64_t(l) * N * KP;
  for (int64_t s0 = n_beg; s0 < n_end; s0 += ST_SUB) {
    __syncthreads();
    for (int e = tid; e < ST_SUB * KP; e += ST_THREADS) {
      const int t = e / KP, s = e % KP;
      xs[t][s] = (s0 + t < n_end) ? Xl[(s0 + t) * KP + s] : 0.f;
    }
    for (int e = tid; e < ST_SUB * C; e += ST_THREADS) {
      const int t = e / C, c = e % C;
      es[t][c] = (s0 + t < n_end) ? E[(s0 + t) * C + c] : 0.f;
    }
    __syncthreads();
#pragma unroll
    for (int i = 0; i < GPT; ++i) {
      const int e = tid + i * ST_THREADS;
      if (e < KP * KP) {
        const int a = e / KP, b = e % KP;
        float acc = 0.f;
#pragma unroll 8
        for (int t = 0; t < ST_SUB; ++t) acc = fmaf(xs[t][a], xs[t][b], acc);
        g[i] += double(acc);
      }
    }
    for (int i = 0; i < SPT; ++i) {
      const int e = tid + i * ST_THREADS;
      if (e < C * KP) {
        const int c = e / KP, s = e % KP;
        float acc = 0.f;
#pragma unroll 8
        for (int t = 0; t < ST_SUB; ++t) acc = fmaf(es[t][c], xs[t][s], acc);
        sacc[i] += double(acc);
      }
    }
    if (tid < ST_SUB) {
      // ||t_n||^2 = u^T (Q Q^T) u with u = e_n P_l
      float u[kMaxRk];
#pragma unroll
      for (int a = 0; a < kMaxRk; ++a) {
        float acc = 0.f;
        if (a < r)
          for (int c = 0; c < C; ++c) acc = fmaf(es[tid][c], Ps[c][a], acc);
        u[a] = acc;
      }
      float qq = 0.f;
#pragma unroll
      for (int a = 0; a < kMaxRk; ++a) {
        if (a >= r) break;
        float mu = 0.f;
#pragma unroll
        for (int b = 0; b < kMaxRk; ++b)
          if (b < r) mu = fmaf(Ms[a][b], u[b], mu);
        qq = fmaf(u[a], mu, qq);
      }
      tq += double(qq);
    }
  }
  const int ps = part_stride(KP, C);
  double* out = part + (int64_t(l) * nch + ch) * ps;
#pragma unroll
  for (int i = 0; i < GPT; ++i) {
    const int e = tid + i * ST_THREADS;
    if (e < KP * KP) out[e] = g[i];
  }
  for (int i = 0; i < SPT; ++i) {
    const int e = tid + i * ST_THREADS;
    if (e < C * KP) out[KP * KP + e] = sacc[i];
  }
  red[tid] = tq;
  __syncthreads();
  for (int w = ST_THREADS / 2; w > 0; w >>= 1) {
    if (tid < w) red[tid] += red[tid + w];
    __syncthreads();
  }
  if (tid == 0) out[ps - 1] = red[0];
}

// ------------------------------------------------------------------ per-block final reduction
constexpr int FI_THREADS = 256;

__global__ void __launch_bounds__(FI_THREADS) k_kspace_final(const double* __restrict__ part,
                                                           const double* __restrict__ xsq_part, int nch,
                                                           int ntiles, int kp, int k, int C, float eta,
                                                           int zero_first, float* __restrict__ G,
                                                           float* __restrict__ SC, double* __restrict__ xsq_total,
                                                           float* __restrict__ alpha_out) {
  __shared__ double red[FI_THREADS];
  __shared__ double s_xsq, s_tsq;
  const int l = blockIdx.x, tid = threadIdx.x;
  const int ps = part_stride(kp, C);
  const double* pl = part + int64_t(l) * nch * ps;
  // xsq of this batch: per-thread strided sums in a fixed order, then a fixed tree
  double a = 0.0;
  for (int64_t i = tid; i < int64_t(ntiles) * 4; i += FI_THREADS) a += xsq_part[int64_t(l) * ntiles * 4 + i];
  red[tid] = a;
  __syncthreads();
  for (int w = FI_THREADS / 2; w > 0; w >>= 1) {
    if (tid < w) red[tid] += red[tid + w];
    __syncthreads();
  }
  if (tid == 0) {
    s_xsq = red[0];
    double t = 0.0;
    for (int c = 0; c < nch; ++c) t += pl[int64_t(c) * ps + ps - 1];
    s_tsq = t;
  }
  __syncthreads();
  const double xsq_b = s_xsq, tsq_b = s_tsq;
  const double al = tsq_b > 0.0 ? -double(eta) * sqrt(xsq_b / tsq_b) : 0.0;
  for (int e = tid; e < k * k; e += FI_THREADS) {
    const int r0 = e / k, c0 = e % k;
    double v = 0.0;
    for (int c = 0; c < nch; ++c) v += pl[int64_t(c) * ps + r0 * kp + c0];
    float* o = G + int64_t(l) * k * k + e;
    *o = zero_first ? float(v) : float(double(*o) + v);
  }
  for (int e = tid; e < C * k; e += FI_THREADS) {
    const int cc = e / k, s = e % k;
    double v = 0.0;
    for (int c = 0; c < nch; ++c) v += pl[int64_t(c) * ps + kp * kp + cc * kp + s];
    float* o = SC + int64_t(l) * C * k + e;
    *o = zero_first ? float(al * v) : float(double(*o) + al * v);
  }
  if (tid == 0) {
    xsq_total[l] = zero_first ? xsq_b : xsq_total[l] + xsq_b;
    if (alpha_out) alpha_out[l] = float(al);
  }
}

// ------------------------------------------------------------------ solve
constexpr int KS_THREADS = 256;

template <int KM>
__global__ void __launch_bounds__(KS_THREADS) k_kspace_solve(
    const float* __restrict__ G, const float* __restrict__ SC, const double* __restrict__ xsq_total,
    const float* __restrict__ P, const float* __restrict__ Q, const float* __restrict__ B_prev, int64_t d,
    int k, int C, int r, int L, float l0, float l1, float l2, float l3, float l4, float l5, float l6, float l7,
    float l8, float l9, float l10, float l11, float l12, float l13, float l14, float l15, float* __restrict__ B,
    int32_t* __restrict__ info, float* __restrict__ C_out) {
  __shared__ float Gf[KM][KM];
  __shared__ double Md[KM][KM];
  __shared__ float Lf[KM][KM];
  __shared__ float Linv[KM];
  __shared__ float W2[kMaxRk][KM];  // P_l^T S_l  (r x k)
  __shared__ int s_info;
  const int j = blockIdx.x, l = blockIdx.y;
  const float lam_rel[16] = {l0, l1, l2, l3, l4, l5, l6, l7, l8, l9, l10, l11, l12, l13, l14, l15};
  for (int e = threadIdx.x; e < KM * KM; e += KS_THREADS) {
    const int a = e / KM, b = e % KM;
    Gf[a][b] = (a < k && b < k) ? G[(int64_t(l) * k + a) * k + b] : 0.f;
  }
  for (int e = threadIdx.x; e < kMaxRk * KM; e += KS_THREADS) {
    const int t = e / KM, s = e % KM;
    float acc = 0.f;
    if (t < r && s < k)
      for (int c = 0; c < C; ++c) acc = fmaf(P[(int64_t(l) * C + c) * r + t], SC[(int64_t(l) * C + c) * k + s], acc);
    W2[t][s] = acc;
  }
  __syncthreads();
  const double lam = double(lam_rel[j]) * (xsq_total != nullptr ? xsq_total[l] / double(d) : 1.0);
  for (int e = threadIdx.x; e < KM * KM; e += KS_THREADS) {
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
  const int inf = chol_factor<KM>(Md, Lf, Linv, &s_info);
  if (threadIdx.x == 0) info[int64_t(j) * L + l] = inf;
  float* Bj = B + (int64_t(j) * L + l) * d * k;
  const float* Bp = B_prev ? B_prev + int64_t(l) * d * k : nullptr;
  const float* Ql = Q + int64_t(l) * r * d;
  for (int64_t i = threadIdx.x; i < d; i += KS_THREADS) {
    float c[KM];
#pragma unroll
    for (int s = 0; s < KM; ++s) c[s] = 0.f;
    for (int t = 0; t < r; ++t) {
      const float qt = Ql[int64_t(t) * d + i];
#pragma unroll
      for (int s = 0; s < KM; ++s) c[s] = fmaf(qt, W2[t][s], c[s]);
    }
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
    if (C_out != nullptr && j == 0) {
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

bool make_map3(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t outer, uint32_t box_rows) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {cuuint64_t(inner), cuuint64_t(rows), cuuint64_t(outer)};
  cuuint64_t strides[2] = {cuuint64_t(inner) * 2, cuuint64_t(rows) * cuuint64_t(inner) * 2};
  cuuint32_t box[3] = {uint32_t(XA_BK), box_rows, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int kp_for(int k) { return k <= 16 ? 16 : 32; }

}  // namespace

// ---- workspace layout (256-byte aligned regions)
KspaceWs kspace_ws(int L, int64_t N, int64_t d, int k, int C, int r) {
  KspaceWs w{};
  const int kp = kp_for(k);
  const int64_t ntiles = (N + XA_TM - 1) / XA_TM;
  const int64_t nch = (N + ST_CHUNK - 1) / ST_CHUNK;
  size_t off = 0;
  w.W = off;
  off += align256(sizeof(__nv_bfloat16) * size_t(L) * 2 * kp * size_t(d));
  w.M = off;
  off += align256(sizeof(float) * size_t(L) * r * r);
  w.Xp = off;
  off += align256(sizeof(float) * size_t(L) * size_t(N) * kp);
  w.xsq_part = off;
  off += align256(sizeof(double) * size_t(L) * size_t(ntiles) * 4);
  w.part = off;
  off += align256(sizeof(double) * size_t(L) * size_t(nch) * part_stride(kp, C));
  w.flags = off;
  off += 256;
  w.total = off;
  return w;
}

int kspace_max_C() { return kMaxCk; }
int kspace_max_r() { return kMaxRk; }

cudaError_t launch_kspace_accumulate(const void* X, int L, int64_t N, int64_t d, const float* A, int k,
                                     const float* E, int C, const float* P, const float* Q, int r, float eta,
                                     int zero_first, float* G, float* SC, double* xsq_total, float* alpha_out,
                                     void* workspace, int32_t* status, cudaStream_t s) {
  const KspaceWs lay = kspace_ws(L, N, d, k, C, r);
  char* ws = static_cast<char*>(workspace);
  __nv_bfloat16* W = reinterpret_cast<__nv_bfloat16*>(ws + lay.W);
  float* M = reinterpret_cast<float*>(ws + lay.M);
  float* Xp = reinterpret_cast<float*>(ws + lay.Xp);
  double* xsq_part = reinterpret_cast<double*>(ws + lay.xsq_part);
  double* part = reinterpret_cast<double*>(ws + lay.part);
  int32_t* abort_flag = reinterpret_cast<int32_t*>(ws + lay.flags);
  const int kp = kp_for(k);
  const int ntiles = int((N + XA_TM - 1) / XA_TM);
  const int nch = int((N + ST_CHUNK - 1) / ST_CHUNK);
  cudaError_t e = cudaMemsetAsync(abort_flag, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  k_kspace_prep<<<dim3(unsigned(L), PREP_SPLIT), PREP_THREADS, 0, s>>>(A, Q, d, k, kp, r, W, M);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  CUtensorMap tmX, tmW;
  if (!make_map3(&tmX, X, uint64_t(d), uint64_t(N), uint64_t(L), XA_TM) ||
      !make_map3(&tmW, W, uint64_t(d), uint64_t(2 * kp), uint64_t(L), uint32_t(2 * kp)))
    return cudaErrorInvalidValue;
  int grid = sm_count();
  if (grid > L * ntiles) grid = L * ntiles;
  const unsigned long long limit = 4000000000ull;
  if (kp == 16) {
    e = cudaFuncSetAttribute(k_kspace_xa<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, XA_SMEM);
    if (e != cudaSuccess) return e;
    k_kspace_xa<16><<<grid, XA_THREADS, XA_SMEM, s>>>(tmX, tmW, L, N, d, ntiles, Xp, xsq_part, status, abort_flag, limit);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_kspace_stats<16><<<dim3(unsigned(nch), unsigned(L)), ST_THREADS, 0, s>>>(Xp, E, P, M, N, C, r, nch, part);
  } else {
    e = cudaFuncSetAttribute(k_kspace_xa<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, XA_SMEM);
    if (e != cudaSuccess) return e;
    k_kspace_xa<32><<<grid, XA_THREADS, XA_SMEM, s>>>(tmX, tmW, L, N, d, ntiles, Xp, xsq_part, status, abort_flag, limit);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_kspace_stats<32><<<dim3(unsigned(nch), unsigned(L)), ST_THREADS, 0, s>>>(Xp, E, P, M, N, C, r, nch, part);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_kspace_final<<<L, FI_THREADS, 0, s>>>(part, xsq_part, nch, ntiles, kp, k, C, eta, zero_first, G, SC, xsq_total,
                                          alpha_out);
  return cudaGetLastError();
}

cudaError_t launch_kspace_solve(const float* G, const float* SC, const double* xsq_total, const float* P,
                                const float* Q, const float* B_prev, const float* lambda_rel, int nl, int L,
                                int64_t d, int k, int C, int r, float* B, int32_t* info, float* C_out,
                                cudaStream_t s) {
  float v[16] = {};
  for (int i = 0; i < nl && i < 16; ++i) v[i] = lambda_rel[i];
  const dim3 grid = dim3(unsigned(nl), unsigned(L));
#define LOCA_KS(KM)                                                                                         \
  k_kspace_solve<KM><<<grid, KS_THREADS, 0, s>>>(G, SC, xsq_total, P, Q, B_prev, d, k, C, r, L, v[0], v[1], \
                                                 v[2], v[3], v[4], v[5], v[6], v[7], v[8], v[9], v[10], v[11], \
                                                 v[12], v[13], v[14], v[15], B, info, C_out)
  if (k <= 4) LOCA_KS(4);
  else if (k <= 8) LOCA_KS(8);
  else if (k <= 16) LOCA_KS(16);
  else LOCA_KS(32);
#undef LOCA_KS
  return cudaGetLastError();
}

}  // namespace loca
