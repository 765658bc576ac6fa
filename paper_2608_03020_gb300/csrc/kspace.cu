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
//   k_kspace_xa     p = W_l x_n on tcgen05 (kind::f16, M = 128 tokens, N = 2 kp, K = 16, both
//                   operands K-major with the 128-byte swizzle): a persistent CTA per SM streams
//                   128-token x 64-channel tiles of X (16 KB) and the matching W tile through an
//                   8-stage TMA ring.  Per tile, four epilogue warps take p = hi part + lo part
//                   from TMEM (one token per thread) and add the tile's sums over their 32 tokens
//                   (p p^T upper triangle, e p^T; fp32) to per-lane registers; each CTA's run of
//                   tiles of a block ends in
//                   one write of its (block, CTA, warp) fp64 partial slot.  Two further warps sum
//                   the squares of every X tile and, with the MMA commit, release the stages, so
//                   the statistics never hold up the ring.  Nothing but X is read from HBM in
//                   bulk, and no warp waits for another outside the mbarrier pipeline.
//   k_kspace_ete    E^T E of the batch (C x C), shared by every block: ||T_l||^2 =
//                   <P_l (Q_l Q_l^T) P_l^T, E^T E>, so no per-token work is needed for it.
//   k_kspace_final  fixed-order reduction of the partial slots per block (deterministic),
//                   ||T_l||^2, alpha_l, and the update of G, S, xsq_total.
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
    const float a = (s < k && LOCA_CHECK(j * k + s, d * k)) ? Al[j * k + s] : 0.f;
    const __nv_bfloat16 hi = __float2bfloat16_rn(a);
    const __nv_bfloat16 lo = __float2bfloat16_rn(a - __bfloat162float(hi));
    if (!LOCA_CHECK(int64_t(kp + s) * d + j, int64_t(2) * kp * d)) continue;
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
    if (lane == 0 && LOCA_CHECK((int64_t(l) * r + a) * r + b, int64_t(gridDim.x) * r * r))
      M[(int64_t(l) * r + a) * r + b] = float(v);
  }
}

// ------------------------------------------------------------------ X A on the tensor cores
// warps: producer, MMA, 4 TMEM / statistics warps, then four sum-of-squares warps, which share the
// 128 token rows of each stage (one row per lane, so that they keep up with the TMA ring) and own
// one of the CTA's four partial slots of ||x||^2 each.  320 threads leave 168 registers a thread.
__host__ __device__ constexpr int xa_sq_warps(int) { return 4; }
__host__ __device__ constexpr int xa_threads(int kp) { return 32 * (6 + xa_sq_warps(kp)); }
static_assert(xa_sq_warps(16) <= 4 && xa_sq_warps(32) <= 4, "four partial slots per CTA");
constexpr int XA_TM = 128;          // tokens per tile (TMEM lanes)
constexpr int XA_BK = 64;           // channels per stage (one 128-byte swizzle row)
constexpr int XA_STAGES = 8;
constexpr int XA_XBYTES = XA_TM * XA_BK * 2;  // 16 KB
constexpr int XA_STAGE = 24 * 1024;           // X tile + up to 64 W rows (8 KB)
constexpr uint32_t XA_TMEM_COLS = 128;
constexpr int XA_MAX_GRID = 256;   // partial slots per block are sized for at most this many CTAs
constexpr int kMaxCk = 16;         // C limit of the k-space path
constexpr int kMaxRk = 32;         // r limit
// per-warp p and e staging: token-major rows at kp = 16 (32 x (33 + 17) floats), channel-major
// rows of 36 floats at kp = 32 ((32 + 16) x 36 floats)
constexpr int XA_EPI_WARP =
    (32 + kMaxCk) * 36 > 32 * (33 + kMaxCk + 1) ? (32 + kMaxCk) * 36 : 32 * (33 + kMaxCk + 1);
constexpr int XA_EPI_SMEM = 4 * XA_EPI_WARP * 4;

// partial slot: upper triangle of p p^T (kp (kp + 1) / 2), e p^T (C x kp), ||x||^2
__host__ __device__ constexpr int ntri(int kp) { return kp * (kp + 1) / 2; }
__host__ __device__ constexpr int part_stride(int kp, int C) { return ntri(kp) + C * kp + 1; }
constexpr int XA_SMEM = XA_STAGES * XA_STAGE + 1024 + 256 + XA_EPI_SMEM;

template <int KP>
__global__ void __launch_bounds__(xa_threads(KP), 1)
    k_kspace_xa(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW, int L,
                int64_t N, int64_t d, int ntiles, const float* __restrict__ E, int C,
                double* __restrict__ part, int32_t* status, int32_t* abort_flag, unsigned long long limit_ns) {
  constexpr int NCOL = 2 * KP;
  constexpr uint32_t WBYTES = uint32_t(NCOL) * 128u;
  constexpr int SQW = xa_sq_warps(KP);
  constexpr int RPW = XA_TM / SQW;  // token rows of a stage per sum-of-squares warp
  constexpr uint32_t ID = tc::idesc(1, 1, 0, 0, XA_TM, NCOL);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + XA_STAGES * XA_STAGE);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * XA_STAGES + 6);
  float* epi = reinterpret_cast<float*>(smem + XA_STAGES * XA_STAGE + 256);
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
      mbar_init(empty_bar(s), 1 + SQW);  // the MMA commit and lane 0 of each sum-of-squares warp
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
          (void)LOCA_REQUIRE((kc * XA_BK) % 8 == 0 && t0 >= 0);
          tma_load_3d(st, &tmX, fb, kc * XA_BK, t0, l);
          tma_load_3d(st + XA_XBYTES, &tmW, fb, kc * XA_BK, 0, l);
          if (++stage == XA_STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        for (int s = 0; s < XA_STAGES; ++s)
          if (pending & (1u << s)) mbar_drain(full_bar(s), (pending_par >> s) & 1u, kDrainLimitNs);
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
        if (!mbar_try_wait(acc_empty(buf), aph ^ 1u) && !mbar_wait(acc_empty(buf), aph ^ 1u, wc)) {
          ok = false;
          break;
        }
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
        mbar_drain(drain_bar, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else if (warp >= 6) {
    // sum-of-squares warps 6..5+SQW: tokens w2 * RPW + h * 32 + lane of every stage; they alone
    // (with the MMA commit) release the stages, so the statistics below never hold up the ring
    const int w2 = warp - 6;
    const int PS = part_stride(KP, C);
    const int64_t nslot = int64_t(gridDim.x) * 4;
    const int xe = ntri(KP) + C * KP;  // the ||x||^2 entry of slots (CTA, w2)
    double xs = 0.0;
    int cur_l = -1;
    auto flush = [&](int lf) {
      double a = xs;
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) a += __shfl_xor_sync(0xffffffffu, a, off);
      if (lane == 0 && LOCA_CHECK((int64_t(lf) * PS + xe) * nslot + int64_t(blockIdx.x) * 4 + w2, int64_t(L) * PS * nslot))
        part[(int64_t(lf) * PS + xe) * nslot + int64_t(blockIdx.x) * 4 + w2] = a;
    };
    int stage = 0;
    uint32_t phase = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x) {
      const int l = it / ntiles;
      if (l != cur_l) {
        if (cur_l >= 0) flush(cur_l);
        cur_l = l;
        xs = 0.0;
      }
      bool ok = true;
      for (int kc = 0; kc < nkc; ++kc) {
        // the bounded wait is a call (registers saved around it): an inline try_wait goes first
        const bool w_ok = mbar_try_wait(full_bar(stage), phase) || mbar_wait(full_bar(stage), phase, wc);
        if (!__all_sync(0xffffffffu, w_ok)) { ok = false; break; }
        // squares of the tokens' 64 channels: rows of the swizzled tile (chunk order is irrelevant
        // for a sum, so lane i starts at chunk i % 8 and the 32 lanes' 16-byte reads spread over
        // all banks); zero-filled out-of-range tokens and channels add nothing
        float pa[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};  // independent chains
#pragma unroll
        for (int h = 0; h < RPW / 32; ++h) {
          const int row = w2 * RPW + h * 32 + lane;
          const uint32_t ra = sbase + uint32_t(stage) * XA_STAGE + uint32_t(row) * 128u;
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            uint32_t w0, w1, w3, w4;
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];" : "=r"(w0), "=r"(w1), "=r"(w3), "=r"(w4)
                         : "r"(ra + uint32_t((c + row) & 7) * 16u));
            const uint32_t wv[4] = {w0, w1, w3, w4};
#pragma unroll
            for (int u = 0; u < 4; ++u) {
              const float lo = __uint_as_float(wv[u] << 16), hi = __uint_as_float(wv[u] & 0xffff0000u);
              pa[2 * u] = fmaf(lo, lo, pa[2 * u]);
              pa[2 * u + 1] = fmaf(hi, hi, pa[2 * u + 1]);
            }
          }
        }
        xs += double(((pa[0] + pa[1]) + (pa[2] + pa[3])) + ((pa[4] + pa[5]) + (pa[6] + pa[7])));
        __syncwarp();
        if (lane == 0) mbar_arrive(empty_bar(stage));
        if (++stage == XA_STAGES) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
    }
    if (cur_l >= 0) flush(cur_l);  // warp-uniform
  } else {
    // epilogue warps 2..5: TMEM lane quarter q; token row = q * 32 + lane of each tile
    const int q = warp & 3;
    const int row = q * 32 + lane;
    constexpr int NTRI = ntri(KP);
    const int PS = part_stride(KP, C);
    constexpr int NSM = (kMaxCk * KP + 31) / 32;
    const int NS = C * KP;
    // p p^T: at kp = 16 a lane owns single upper-triangle entries eidx = lane + 32 i; at kp = 32
    // it owns 2 x 2 blocks (rows 2I, 2I+1; columns 2J, 2J+1; I <= J) of the 16 x 16 block
    // triangle, bidx = lane + 32 i, whose p rows it reads four tokens at a time.  Either way each
    // entry is the same fp32 FMA chain over the tile's tokens in order.
    constexpr bool kBlk = KP > 16;
    constexpr int KQ = kBlk ? KP / 2 : KP;   // side of the triangle a lane's items tile
    constexpr int NQ = ntri(KQ);
    constexpr int NG = (NQ + 31) / 32;
    constexpr int NACC = kBlk ? 4 * NG : NG;
    // item lane + 32 i -> (a, b), row-major over the triangle: (a << 8) | b at kp = 16; at kp = 32
    // (a, b < 16) packed as (a << 4) | b into byte i % 4 of word i / 4
    constexpr int NPW = kBlk ? (NG + 3) / 4 : NG;
    uint32_t pair[NPW];
#pragma unroll
    for (int i2 = 0; i2 < NPW; ++i2) pair[i2] = 0u;
#pragma unroll
    for (int i2 = 0; i2 < NG; ++i2) {
      int rem = lane + 32 * i2, a = 0;
      while (a < KQ && rem >= KQ - a) {
        rem -= KQ - a;
        ++a;
      }
      if constexpr (kBlk)
        pair[i2 / 4] |= uint32_t(((a << 4) | ((a + rem) & 15)) & 0xff) << (8 * (i2 % 4));
      else
        pair[i2] = uint32_t((a << 8) | (a + rem));
    }
    auto blk_pair = [&](int i2, int& bi, int& bj) {
      const uint32_t x = (pair[i2 / 4] >> (8 * (i2 % 4))) & 0xffu;
      bi = int(x >> 4);
      bj = int(x & 15u);
    };
    // staging.  kp = 16: token-major rows (ps[t][s], es[t][c]).  kp = 32: channel-major rows of
    // 36 floats (pT[.][t], eT[c][t]; 16-byte aligned for four-token loads), p row s stored at
    // (s / 2) + 16 (s % 2) so that the column rows 2J of eight lanes fall in distinct banks.
    constexpr int PSTR = KP + 1, ESTR = kMaxCk + 1;
    constexpr int TST = 36;
    float* ps = epi + (warp - 2) * (kBlk ? (32 + kMaxCk) * TST : 32 * (33 + ESTR));
    float* es = kBlk ? ps + 32 * TST : ps + 32 * 33;
    auto prow = [](int s2) { return (s2 >> 1) + (s2 & 1) * (KP / 2); };
    auto entry = [](int a, int b) { return a * KP - a * (a - 1) / 2 + (b - a); };
    // this lane's sums for the current block (fp32 within one CTA's run of tiles of a block; the
    // runs are written once, as fp64, when the block changes, and reduced in a fixed order later)
    float accg[NACC], accs[NSM];
    int cur_l = -1;
    const int64_t nslot = int64_t(gridDim.x) * 4;
    auto flush = [&](int lf) {
      // entry-major: entry e of block lf at part[(lf * PS + e) * nslot + this slot]
      double* slot = part + int64_t(lf) * PS * nslot + int64_t(blockIdx.x) * 4 + q;
      // every entry index below is < PS - 1 (the last one is the ||x||^2 entry of the other warps)
      if (!LOCA_CHECK(lf, L) || !LOCA_REQUIRE(NTRI + NS + 1 == PS)) return;
      if constexpr (kBlk) {
#pragma unroll
        for (int i2 = 0; i2 < NG; ++i2) {
          if (lane + 32 * i2 < NQ) {
            int bi, bj;
            blk_pair(i2, bi, bj);
            const int a0 = 2 * bi, b0 = 2 * bj;
            slot[int64_t(entry(a0, b0)) * nslot] = double(accg[4 * i2]);
            slot[int64_t(entry(a0, b0 + 1)) * nslot] = double(accg[4 * i2 + 1]);
            if (a0 != b0) slot[int64_t(entry(a0 + 1, b0)) * nslot] = double(accg[4 * i2 + 2]);
            slot[int64_t(entry(a0 + 1, b0 + 1)) * nslot] = double(accg[4 * i2 + 3]);
          }
        }
      } else {
#pragma unroll
        for (int i2 = 0; i2 < NG; ++i2)
          if (lane + 32 * i2 < NTRI) slot[int64_t(lane + 32 * i2) * nslot] = double(accg[i2]);
      }
#pragma unroll
      for (int i2 = 0; i2 < NSM; ++i2)
        if (lane + 32 * i2 < NS) slot[int64_t(NTRI + lane + 32 * i2) * nslot] = double(accs[i2]);
    };
    uint32_t tcount = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x, ++tcount) {
      const int l = it / ntiles;
      const int tile = it - l * ntiles;
      const int t0 = tile * XA_TM;
      if (l != cur_l) {
        if (cur_l >= 0) flush(cur_l);
        cur_l = l;
#pragma unroll
        for (int i2 = 0; i2 < NACC; ++i2) accg[i2] = 0.f;
#pragma unroll
        for (int i2 = 0; i2 < NSM; ++i2) accs[i2] = 0.f;
      }
      const int buf = int(tcount & 1u);
      const uint32_t aph = (tcount >> 1) & 1u;
      const bool a_ok = mbar_try_wait(acc_full(buf), aph) || mbar_wait(acc_full(buf), aph, wc);
      if (!__all_sync(0xffffffffu, a_ok)) break;
      fence_after();
      const uint32_t ta = tmem_base + (uint32_t(q * 32) << 16) + uint32_t(buf * NCOL);
      // stage this warp's 32 tokens: p (kp) and e (C); tokens beyond N contribute zeros.  p is the
      // sum of the hi and lo accumulator columns; at kp = 32 the two halves are read one after the
      // other (hi staged, then lo added to it: the same fp32 sum)
      if constexpr (kBlk) {
        const int64_t n = int64_t(t0) + row;
        const bool nv = n < N;
        float v[32];
        tmem_ld32(ta, v);
#pragma unroll
        for (int s2 = 0; s2 < KP; ++s2) ps[prow(s2) * TST + lane] = v[s2];
        tmem_ld32(ta + uint32_t(KP), v);
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty(buf));
#pragma unroll
        for (int s2 = 0; s2 < KP; ++s2) {
          float* d = ps + prow(s2) * TST + lane;
          *d = *d + v[s2];
        }
#pragma unroll
        for (int c = 0; c < kMaxCk; ++c)
          if (c < C) es[c * TST + lane] = (nv && LOCA_CHECK(n * C + c, N * C)) ? E[n * C + c] : 0.f;
      } else {
        float v[NCOL];
        if constexpr (NCOL == 32) {
          tmem_ld32(ta, v);
        } else {
          tmem_ld32x2(ta, v);
        }
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty(buf));
        const int64_t n = int64_t(t0) + row;
        const bool nv = n < N;
#pragma unroll
        for (int s2 = 0; s2 < KP; ++s2) ps[lane * PSTR + s2] = v[s2] + v[KP + s2];
#pragma unroll
        for (int c = 0; c < kMaxCk; ++c)
          if (c < C) es[lane * ESTR + c] = (nv && LOCA_CHECK(n * C + c, N * C)) ? E[n * C + c] : 0.f;
      }
      __syncwarp();
      // the tile's sums over this warp's 32 tokens, for the entries this lane owns
      if constexpr (kBlk) {
#pragma unroll
        for (int i2 = 0; i2 < NG; ++i2) {
          if (lane + 32 * i2 < NQ) {
            int bi, bj;
            blk_pair(i2, bi, bj);
            const float* ra0 = ps + prow(2 * bi) * TST;
            const float* ra1 = ps + prow(2 * bi + 1) * TST;
            const float* rb0 = ps + prow(2 * bj) * TST;
            const float* rb1 = ps + prow(2 * bj + 1) * TST;
            float s00 = 0.f, s01 = 0.f, s10 = 0.f, s11 = 0.f;
#pragma unroll 2
            for (int t = 0; t < 32; t += 4) {
              const float4 x0 = *reinterpret_cast<const float4*>(ra0 + t);
              const float4 x1 = *reinterpret_cast<const float4*>(ra1 + t);
              const float4 y0 = *reinterpret_cast<const float4*>(rb0 + t);
              const float4 y1 = *reinterpret_cast<const float4*>(rb1 + t);
              s00 = fmaf(x0.x, y0.x, s00); s01 = fmaf(x0.x, y1.x, s01);
              s10 = fmaf(x1.x, y0.x, s10); s11 = fmaf(x1.x, y1.x, s11);
              s00 = fmaf(x0.y, y0.y, s00); s01 = fmaf(x0.y, y1.y, s01);
              s10 = fmaf(x1.y, y0.y, s10); s11 = fmaf(x1.y, y1.y, s11);
              s00 = fmaf(x0.z, y0.z, s00); s01 = fmaf(x0.z, y1.z, s01);
              s10 = fmaf(x1.z, y0.z, s10); s11 = fmaf(x1.z, y1.z, s11);
              s00 = fmaf(x0.w, y0.w, s00); s01 = fmaf(x0.w, y1.w, s01);
              s10 = fmaf(x1.w, y0.w, s10); s11 = fmaf(x1.w, y1.w, s11);
            }
            accg[4 * i2] += s00;
            accg[4 * i2 + 1] += s01;
            accg[4 * i2 + 2] += s10;
            accg[4 * i2 + 3] += s11;
          }
        }
        // e p^T: this lane's channel s = lane of every label column c (eidx = c kp + lane)
        const float* rp = ps + prow(lane) * TST;
        static_assert(!kBlk || NSM == kMaxCk, "one e p^T entry per label column and lane");
#pragma unroll
        for (int c = 0; c < kMaxCk; ++c) {
          if (c < C) {
            const float* re = es + c * TST;
            float sc = 0.f;
#pragma unroll 1
            for (int t = 0; t < 32; t += 4) {
              const float4 pv = *reinterpret_cast<const float4*>(rp + t);
              const float4 ev = *reinterpret_cast<const float4*>(re + t);
              sc = fmaf(ev.x, pv.x, sc);
              sc = fmaf(ev.y, pv.y, sc);
              sc = fmaf(ev.z, pv.z, sc);
              sc = fmaf(ev.w, pv.w, sc);
            }
            accs[c] += sc;
          }
        }
      } else {
#pragma unroll
        for (int i2 = 0; i2 < NG; ++i2) {
          if (lane + 32 * i2 < NTRI) {
            const int a = int(pair[i2] >> 8), b = int(pair[i2] & 0xffu);
            float acc = 0.f;
#pragma unroll 8
            for (int t = 0; t < 32; ++t) acc = fmaf(ps[t * PSTR + a], ps[t * PSTR + b], acc);
            accg[i2] += acc;
          }
        }
#pragma unroll
        for (int i2 = 0; i2 < NSM; ++i2) {
          const int eidx = lane + 32 * i2;
          if (eidx < NS) {
            const int c = eidx / KP, s2 = eidx - c * KP;
            float acc = 0.f;
#pragma unroll 8
            for (int t = 0; t < 32; ++t) acc = fmaf(es[t * ESTR + c], ps[t * PSTR + s2], acc);
            accs[i2] += acc;
          }
        }
      }
      __syncwarp();  // the staging rows are rewritten by the next tile
    }
    if (cur_l >= 0) flush(cur_l);  // warp-uniform: every lane reaches here together
  }

  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, XA_TMEM_COLS);
}

// ------------------------------------------------------------------ E^T E
// ||T_l||^2 = sum_n u_n^T (Q_l Q_l^T) u_n = <P_l (Q_l Q_l^T) P_l^T, E^T E>: the C x C matrix E^T E
// of the batch serves every block.  Partials per chunk of tokens (fp32 over 256 tokens, fp64
// across), reduced in a fixed order by k_kspace_final.
constexpr int ETE_THREADS = 256;
constexpr int ETE_SUB = 256;
constexpr int ETE_CHUNK = 1024;

__global__ void __launch_bounds__(ETE_THREADS) k_kspace_ete(const float* __restrict__ E, int64_t N, int C,
                                                          double* __restrict__ ete_part) {
  __shared__ float es[ETE_SUB][kMaxCk + 1];
  const int ch = blockIdx.x, tid = threadIdx.x;
  const int a = tid / kMaxCk, b = tid % kMaxCk;
  const int64_t n0 = int64_t(ch) * ETE_CHUNK;
  const int64_t n1 = (n0 + ETE_CHUNK < N) ? n0 + ETE_CHUNK : N;
  double acc = 0.0;
  for (int64_t s0 = n0; s0 < n1; s0 += ETE_SUB) {
    __syncthreads();
    for (int e = tid; e < ETE_SUB * C; e += ETE_THREADS) {
      const int t = e / C, c = e % C;
      es[t][c] = (s0 + t < n1 && LOCA_CHECK((s0 + t) * C + c, N * C)) ? E[(s0 + t) * C + c] : 0.f;
    }
    __syncthreads();
    if (a < C && b < C) {
      float part = 0.f;
#pragma unroll 8
      for (int t = 0; t < ETE_SUB; ++t) part = fmaf(es[t][a], es[t][b], part);
      acc += double(part);
    }
  }
  if (a < C && b < C && LOCA_CHECK(int64_t(ch) * kMaxCk * kMaxCk + a * kMaxCk + b, int64_t(gridDim.x) * kMaxCk * kMaxCk))
    ete_part[int64_t(ch) * kMaxCk * kMaxCk + a * kMaxCk + b] = acc;
}

// ------------------------------------------------------------------ per-block final reduction
constexpr int FI_THREADS = 256;
constexpr int FI_SPLIT = 4;  // CTAs per block (entries e with e % FI_SPLIT == part)

// Sums the (CTA, warp) partial slots of block l in a fixed order (a CTA without tiles of block l,
// possible only when blocks have fewer tiles than there are CTAs, never wrote its slot), forms
// ||T_l||^2 = <P_l M_l P_l^T, E^T E>, the step alpha_l, and updates G, SC, xsq_total.
__global__ void __launch_bounds__(FI_THREADS) k_kspace_final(const double* __restrict__ part,
                                                           const double* __restrict__ ete_part, int nch_e,
                                                           const float* __restrict__ P, const float* __restrict__ M,
                                                           int grid, int ntiles, int kp, int k, int C, int r,
                                                           float eta, int zero_first, float* __restrict__ G,
                                                           float* __restrict__ SC, double* __restrict__ xsq_total,
                                                           float* __restrict__ alpha_out) {
  __shared__ unsigned char has[XA_MAX_GRID];
  __shared__ double ete[kMaxCk][kMaxCk];
  __shared__ double pm[kMaxCk][kMaxRk];  // P_l M_l
  __shared__ double red[FI_THREADS];
  __shared__ double s_xsq;
  const int l = blockIdx.x, prt = blockIdx.y, tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ps = part_stride(kp, C);
  const int64_t lo = int64_t(l) * ntiles, hi = lo + ntiles;
  for (int c = tid; c < grid; c += FI_THREADS) has[c] = (lo + ((int64_t(c) - lo) % grid + grid) % grid) < hi;
  for (int e = tid; e < C * C; e += FI_THREADS) {
    const int a = e / C, b = e % C;
    double v = 0.0;
    for (int ch = 0; ch < nch_e; ++ch) v += ete_part[int64_t(ch) * kMaxCk * kMaxCk + a * kMaxCk + b];
    ete[a][b] = v;
  }
  const float* Pl = P + int64_t(l) * C * r;
  const float* Ml = M + int64_t(l) * r * r;
  for (int e = tid; e < C * r; e += FI_THREADS) {
    const int c = e / r, b = e % r;
    double v = 0.0;
    for (int a = 0; a < r; ++a) v += double(Pl[c * r + a]) * double(Ml[a * r + b]);
    pm[c][b] = v;
  }
  __syncthreads();
  const int nslot = grid * 4;
  // one warp; lanes over slots in order, then a fixed butterfly.  The ||x||^2 entry is written
  // by the sum-of-squares warps, one slot each (slots 0..xa_sq_warps(kp)-1 of each CTA).
  auto sum_entry = [&](int e, int nq) {
    const double* pe = part + (int64_t(l) * ps + e) * nslot;
    double v = 0.0;
    for (int sidx = lane; sidx < nslot; sidx += 32)
      if (has[sidx >> 2] && (sidx & 3) < nq) v += pe[sidx];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
    return v;
  };
  const int nt = ntri(kp);
  if (warp == 0) {
    const double v = sum_entry(nt + C * kp, xa_sq_warps(kp));
    if (lane == 0) s_xsq = v;
  }
  // ||T_l||^2 = sum_{c, c'} (P M P^T)[c][c'] (E^T E)[c][c']
  double t = 0.0;
  for (int e = tid; e < C * C; e += FI_THREADS) {
    const int a = e / C, b = e % C;
    double kab = 0.0;
    for (int j = 0; j < r; ++j) kab += pm[a][j] * double(Pl[b * r + j]);
    t += kab * ete[a][b];
  }
  red[tid] = t;
  __syncthreads();
  for (int w = FI_THREADS / 2; w > 0; w >>= 1) {
    if (tid < w) red[tid] += red[tid + w];
    __syncthreads();
  }
  const double xsq_b = s_xsq, tsq_b = red[0];
  const double al = tsq_b > 0.0 ? -double(eta) * sqrt(xsq_b / tsq_b) : 0.0;
  // G entries (symmetric, from the upper triangle) and SC entries of this CTA's share
  for (int e = prt * (FI_THREADS / 32) + warp; e < k * k + C * k; e += FI_SPLIT * (FI_THREADS / 32)) {
    if (e < k * k) {
      int a = e / k, b = e % k;
      if (a > b) {
        const int tmp = a;
        a = b;
        b = tmp;
      }
      const double v = sum_entry(a * kp - a * (a - 1) / 2 + (b - a), 4);  // row a of the upper triangle
      if (lane == 0 && LOCA_CHECK(int64_t(l) * k * k + e, int64_t(gridDim.x) * k * k)) {
        float* o = G + int64_t(l) * k * k + e;
        *o = zero_first ? float(v) : float(double(*o) + v);
      }
    } else {
      const int e2 = e - k * k;
      const int cc = e2 / k, s2 = e2 % k;
      const double v = sum_entry(nt + cc * kp + s2, 4);
      if (lane == 0 && LOCA_CHECK(int64_t(l) * C * k + e2, int64_t(gridDim.x) * C * k)) {
        float* o = SC + int64_t(l) * C * k + e2;
        *o = zero_first ? float(al * v) : float(double(*o) + al * v);
      }
    }
  }
  if (prt == 0 && tid == 0 && LOCA_CHECK(l, gridDim.x)) {
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
  if (threadIdx.x == 0 && LOCA_CHECK(int64_t(j) * L + l, int64_t(gridDim.x) * L)) info[int64_t(j) * L + l] = inf;
  float* Bj = B + (int64_t(j) * L + l) * d * k;
  const float* Bp = B_prev ? B_prev + int64_t(l) * d * k : nullptr;
  const float* Ql = Q + int64_t(l) * r * d;
  for (int64_t i = threadIdx.x; i < d; i += KS_THREADS) {
    if (!LOCA_CHECK_SPAN((int64_t(j) * L + l) * d * k + i * k, k, int64_t(gridDim.x) * L * d * k) ||
        !LOCA_CHECK_SPAN((int64_t(l) * d + i) * k, k, int64_t(L) * d * k))
      break;
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
  size_t off = 0;
  w.W = off;
  off += align256(sizeof(__nv_bfloat16) * size_t(L) * 2 * kp * size_t(d));
  w.M = off;
  off += align256(sizeof(float) * size_t(L) * r * r);
  w.part = off;
  off += align256(sizeof(double) * size_t(L) * XA_MAX_GRID * 4 * part_stride(kp, C));
  w.ete = off;
  off += align256(sizeof(double) * size_t((N + ETE_CHUNK - 1) / ETE_CHUNK) * kMaxCk * kMaxCk);
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
  double* part = reinterpret_cast<double*>(ws + lay.part);
  double* ete = reinterpret_cast<double*>(ws + lay.ete);
  int32_t* abort_flag = reinterpret_cast<int32_t*>(ws + lay.flags);
  const int kp = kp_for(k);
  const int ntiles = int((N + XA_TM - 1) / XA_TM);
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
  if (grid > XA_MAX_GRID) grid = XA_MAX_GRID;
  if (grid > L * ntiles) grid = L * ntiles;
  const unsigned long long limit = wait_limit_ns();
  if (kp == 16) {
    e = cudaFuncSetAttribute(k_kspace_xa<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, XA_SMEM);
    if (e != cudaSuccess) return e;
    k_kspace_xa<16><<<grid, xa_threads(16), XA_SMEM, s>>>(tmX, tmW, L, N, d, ntiles, E, C, part, status,
                                                            abort_flag, limit);
  } else {
    e = cudaFuncSetAttribute(k_kspace_xa<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, XA_SMEM);
    if (e != cudaSuccess) return e;
    k_kspace_xa<32><<<grid, xa_threads(32), XA_SMEM, s>>>(tmX, tmW, L, N, d, ntiles, E, C, part, status,
                                                            abort_flag, limit);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int nch_e = int((N + ETE_CHUNK - 1) / ETE_CHUNK);
  k_kspace_ete<<<nch_e, ETE_THREADS, 0, s>>>(E, N, C, ete);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  k_kspace_final<<<dim3(unsigned(L), FI_SPLIT), FI_THREADS, 0, s>>>(part, ete, nch_e, P, M, grid, ntiles, kp, k, C,
                                                                     r, eta, zero_first, G, SC, xsq_total, alpha_out);
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
