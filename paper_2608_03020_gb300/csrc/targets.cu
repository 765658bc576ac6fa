// Tokenwise feedback predictions of every block (S3: Q_l := F_l E), applied through the
// low-rank factors (S11: F e = U_k (S_k (V_k^T e))):  T_l = (E P_l) Q_l,  on the tensor cores.
//
// The product U Q_l has inner dimension r (4..32), so it is a short tcgen05 MMA per output
// tile; the kernel is bound by the HBM write of T (2 bytes per element in bf16).  Precision:
// U and Q are split into tf32 pairs (hi = rna(x), lo = rna(x - hi)) and the tile is
// hi*hi + hi*lo + lo*hi with fp32 accumulation (kind::tf32), ~2^-20 relative per product, so
// the fp32 output matches an fp32 FMA evaluation.
//
// Persistent, one CTA per SM, 288 threads:
//   warps 0-3   producers: per item load Q_l[:, 256-channel tile], split it into hi/lo K-major
//               tiles (B); per 128-token tile, thread i forms u = E[n0 + i] P_l (fp32), splits
//               it and writes its row of the A tiles (double-buffered).
//   warp 8      owns 512 TMEM columns (two 128 x 256 fp32 accumulators) and issues the MMAs.
//   warps 4-7   epilogue: tcgen05.ld, sum of squares of the fp32 values (||T_l||^2), rounding
//               to the output type; in bf16 each warp stages its 32 token rows in shared
//               memory (128-byte swizzled boxes) and writes them with TMA bulk tensor stores
//               (two 128-channel boxes per tile when d % 64 == 0), so HBM sees whole lines;
//               fp32 output uses plain stores (one row per thread).  TMEM is read 64 columns
//               per wait.
// Work item = (block l, 256-channel tile, 4096-token chunk); ||T_l||^2 partials are written
// per item and epilogue warp and summed in a fixed order by k_reduce_partials
// (deterministic).  All waits are bounded (see tc_ptx.cuh) and no warp waits on another
// warp except through those bounded mbarrier waits.
#include <cuda_bf16.h>

#include <cstring>

#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

using namespace tc;

constexpr int TM = 128;           // tokens per tile (TMEM lanes)
constexpr int TCH = 256;          // channels per tile (TMEM columns per accumulator)
constexpr int CHUNK_TILES = 32;   // tiles per work item
constexpr int CHUNK = TM * CHUNK_TILES;
constexpr int kMaxC = 64;
constexpr int kMaxRP = 32;        // padded feedback rank (multiple of 8)
constexpr int NTHREADS = 288;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t ID_TF32 = idesc(2, 2, 0, 0, TM, TCH);

constexpr uint32_t STAGE_WARP = 32 * TCH * 2;  // one epilogue warp's 32 x 256 bf16 rows (16 KB)

struct Layout {
  uint32_t stage, b_hi, b_lo, a_hi[2], a_lo[2], bars, total;
};
__host__ __device__ inline Layout layout_for(int rp) {
  Layout o;
  const uint32_t b = uint32_t(TCH) * rp * 4, a = uint32_t(TM) * rp * 4;
  o.stage = 0;  // 4 x 16 KB, 1024-byte aligned (128-byte swizzled TMA boxes)
  const uint32_t base = 4 * STAGE_WARP;
  o.b_hi = base;
  o.b_lo = base + b;
  o.a_hi[0] = base + 2 * b;
  o.a_lo[0] = base + 2 * b + a;
  o.a_hi[1] = base + 2 * b + 2 * a;
  o.a_lo[1] = base + 2 * b + 3 * a;
  o.bars = base + 2 * b + 4 * a;
  o.total = o.bars + 256 + 1024;  // + alignment slack
  // at least 120 KB so that one CTA (which takes all 512 TMEM columns) sits on each SM
  if (o.total < 120u * 1024u) o.total = 120u * 1024u;
  return o;
}

// byte offset of element (row m, k s) in a K-major, no-swizzle canonical tile with rp columns:
// 8-row x 16-byte core matrices, K-adjacent ones 128 bytes apart, 8-row groups rp*32 bytes apart
__device__ __forceinline__ uint32_t kmaj_off(int m, int s, int rp) {
  return uint32_t(m >> 3) * uint32_t(rp * 32) + uint32_t(s >> 2) * 128u + uint32_t(m & 7) * 16u +
         uint32_t(s & 3) * 4u;
}

__device__ __forceinline__ uint32_t tf32_rna(float x) {
  uint32_t y;
  asm("cvt.rna.tf32.f32 %0, %1;" : "=r"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

struct Geo {
  int64_t N, d;
  int C, r, rp, L;
  int64_t nd, nchunks, items;
};

__device__ __forceinline__ void decode(const Geo& g, int64_t it, int& l, int64_t& jt, int64_t& ck) {
  l = int(it / (g.nd * g.nchunks));
  const int64_t rem = it - int64_t(l) * g.nd * g.nchunks;
  jt = rem / g.nchunks;
  ck = rem - jt * g.nchunks;
}

template <bool kBF16>
__global__ void __launch_bounds__(NTHREADS, 1)
    k_targets_tc(const float* __restrict__ E, const float* __restrict__ P, const float* __restrict__ Q,
                 Geo g, void* __restrict__ Tout, const __grid_constant__ CUtensorMap tmT, int store_mode,
                 double* __restrict__ partials, int32_t* status, int32_t* abort_flag,
                 unsigned long long limit_ns) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  // 1024-byte aligned base: the 128-byte swizzle of the TMA boxes repeats every 1024 bytes
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const Layout lay = layout_for(g.rp);
  const uint32_t sbase = smem_u32(smem);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + lay.bars);
  // bars: a_full[2], a_empty[2], acc_full[2], acc_empty[2], b_full, b_empty, drain
  const uint32_t bar0 = smem_u32(bars);
  auto a_full = [&](int b) { return bar0 + 8u * b; };
  auto a_empty = [&](int b) { return bar0 + 8u * (2 + b); };
  auto acc_full = [&](int b) { return bar0 + 8u * (4 + b); };
  auto acc_empty = [&](int b) { return bar0 + 8u * (6 + b); };
  const uint32_t b_full = bar0 + 64, b_empty = bar0 + 72, drain_bar = bar0 + 80;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 11);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{status, abort_flag, limit_ns};
  const int rp = g.rp, r = g.r, C = g.C;

  if (threadIdx.x == 0) {
    for (int b = 0; b < 2; ++b) {
      mbar_init(a_full(b), 128);
      mbar_init(a_empty(b), 1);
      mbar_init(acc_full(b), 1);
      mbar_init(acc_empty(b), 128);
    }
    mbar_init(b_full, 128);
    mbar_init(b_empty, 1);
    mbar_init(drain_bar, 1);
    mbar_init_fence();
  }
  if (warp == 8) tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp < 4) {
    // ---------------- producers: thread i <-> tile row i
    const int i = threadIdx.x;
    uint32_t tcount = 0, icount = 0;
    bool ok = true;
    for (int64_t it = blockIdx.x; it < g.items && ok; it += gridDim.x, ++icount) {
      int l;
      int64_t jt, ck;
      decode(g, it, l, jt, ck);
      const int64_t j0 = jt * TCH;
      const int64_t nbeg = ck * CHUNK;
      const int64_t nend = (nbeg + CHUNK < g.N) ? nbeg + CHUNK : g.N;
      // the bounded waits are calls (registers saved around them): an inline try_wait goes first
      if (!mbar_try_wait(b_empty, (icount & 1u) ^ 1u) && !mbar_wait(b_empty, (icount & 1u) ^ 1u, wc)) {
        ok = false;
        break;
      }
      // B = Q_l[:, j0 : j0 + 256] as hi/lo K-major tiles (channel = row, s = k)
      const float* Ql = Q + int64_t(l) * r * g.d;
      for (int h = 0; h < 2; ++h) {
        const int j = i + 128 * h;
        const bool jv = j0 + j < g.d;
        for (int s4 = 0; s4 < rp; s4 += 4) {
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const int s = s4 + u;
            const float x = (jv && s < r && LOCA_CHECK(int64_t(l) * r * g.d + int64_t(s) * g.d + j0 + j,
                                                       int64_t(g.L) * r * g.d))
                                ? Ql[int64_t(s) * g.d + j0 + j]
                                : 0.f;
            hi[u] = tf32_rna(x);
            lo[u] = tf32_rna(x - __uint_as_float(hi[u]));
          }
          const uint32_t off = kmaj_off(j, s4, rp);
          if (!LOCA_CHECK_SPAN(off, 16, uint32_t(TCH) * rp * 4)) continue;
          *reinterpret_cast<uint4*>(smem + lay.b_hi + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(smem + lay.b_lo + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
      }
      fence_proxy_async_smem();
      mbar_arrive(b_full);
      const float* Pl = P + int64_t(l) * C * r;  // read by every producer thread (cached)
      for (int64_t n0 = nbeg; n0 < nend; n0 += TM, ++tcount) {
        const int buf = int(tcount & 1u);
        const uint32_t ph = (tcount >> 1) & 1u;
        const int64_t n = n0 + i;
        float u[kMaxRP];
#pragma unroll
        for (int s = 0; s < kMaxRP; ++s) u[s] = 0.f;
        if (n < nend && LOCA_CHECK_SPAN(n * C, C, g.N * C) && LOCA_CHECK_SPAN(int64_t(l) * C * r, C * r, int64_t(g.L) * C * r)) {
          const float* er = E + n * C;
          for (int c = 0; c < C; ++c) {
            const float ec = er[c];
            const float* pr = Pl + c * r;
#pragma unroll
            for (int s = 0; s < kMaxRP; ++s)
              if (s < r) u[s] = fmaf(ec, __ldg(pr + s), u[s]);
          }
        }
        if (!mbar_try_wait(a_empty(buf), ph ^ 1u) && !mbar_wait(a_empty(buf), ph ^ 1u, wc)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int s4 = 0; s4 < kMaxRP; s4 += 4) {
          if (s4 >= rp) break;
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int v = 0; v < 4; ++v) {
            hi[v] = tf32_rna(u[s4 + v]);
            lo[v] = tf32_rna(u[s4 + v] - __uint_as_float(hi[v]));
          }
          const uint32_t off = kmaj_off(i, s4, rp);
          if (!LOCA_CHECK_SPAN(off, 16, uint32_t(TM) * rp * 4)) continue;
          *reinterpret_cast<uint4*>(smem + lay.a_hi[buf] + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(smem + lay.a_lo[buf] + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
        fence_proxy_async_smem();
        mbar_arrive(a_full(buf));
      }
    }
  } else if (warp == 8) {
    // ---------------- MMA issuer
    if (lane == 0) {
      uint32_t tcount = 0, icount = 0;
      bool ok = true, issued = false;
      const uint32_t sbo = uint32_t(rp) * 32u;
      for (int64_t it = blockIdx.x; it < g.items && ok; it += gridDim.x, ++icount) {
        int l;
        int64_t jt, ck;
        decode(g, it, l, jt, ck);
        const int64_t nbeg = ck * CHUNK;
        const int64_t nend = (nbeg + CHUNK < g.N) ? nbeg + CHUNK : g.N;
        if (!mbar_try_wait(b_full, icount & 1u) && !mbar_wait(b_full, icount & 1u, wc)) {
          ok = false;
          break;
        }
        fence_after();
        for (int64_t n0 = nbeg; n0 < nend; n0 += TM, ++tcount) {
          const int buf = int(tcount & 1u);
          const uint32_t ph = (tcount >> 1) & 1u;
          if ((!mbar_try_wait(acc_empty(buf), ph ^ 1u) && !mbar_wait(acc_empty(buf), ph ^ 1u, wc)) ||
              (!mbar_try_wait(a_full(buf), ph) && !mbar_wait(a_full(buf), ph, wc))) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t d_tmem = tmem_base + uint32_t(buf) * TCH;
          for (int kk = 0; kk < rp / 8; ++kk) {
            const uint32_t koff = uint32_t(kk) * 256u;  // 8 k = two core matrices
            const uint64_t ah = sdesc(sbase + lay.a_hi[buf] + koff, 128u, sbo, kSwizzleNone);
            const uint64_t al = sdesc(sbase + lay.a_lo[buf] + koff, 128u, sbo, kSwizzleNone);
            const uint64_t bh = sdesc(sbase + lay.b_hi + koff, 128u, sbo, kSwizzleNone);
            const uint64_t bl = sdesc(sbase + lay.b_lo + koff, 128u, sbo, kSwizzleNone);
            mma_tf32(d_tmem, ah, bh, ID_TF32, kk > 0 ? 1u : 0u);
            mma_tf32(d_tmem, ah, bl, ID_TF32, 1u);
            mma_tf32(d_tmem, al, bh, ID_TF32, 1u);
          }
          issued = true;
          mma_commit(a_empty(buf));
          mma_commit(acc_full(buf));
        }
        if (!ok) break;
        mma_commit(b_empty);
      }
      if (!ok && issued) {
        mma_commit(drain_bar);
        mbar_drain(drain_bar, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 4..7, TMEM lane quarter = warp % 4
    const int q = warp & 3;
    const int row = q * 32 + lane;
    uint32_t tcount = 0;
    bool ok = true;
    for (int64_t it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
      int l;
      int64_t jt, ck;
      decode(g, it, l, jt, ck);
      const int64_t j0 = jt * TCH;
      const int64_t nbeg = ck * CHUNK;
      const int64_t nend = (nbeg + CHUNK < g.N) ? nbeg + CHUNK : g.N;
      float sq = 0.f;
      double sqd = 0.0;
      for (int64_t n0 = nbeg; n0 < nend; n0 += TM, ++tcount) {
        const int buf = int(tcount & 1u);
        const uint32_t ph = (tcount >> 1) & 1u;
        const bool w_ok = mbar_try_wait(acc_full(buf), ph) || mbar_wait(acc_full(buf), ph, wc);
        if (!__all_sync(0xffffffffu, w_ok)) { ok = false; break; }
        fence_after();
        const int64_t n = n0 + row;
        const bool nv = n < nend;
        const int64_t rbase = (int64_t(l) * g.N + n) * g.d;
        const uint32_t stage = sbase + lay.stage + uint32_t(q) * STAGE_WARP;
#pragma unroll 1
        for (int cp = 0; cp < TCH / 64; ++cp) {
          // 64 channels (one 128-byte swizzled box) per step; two TMEM loads, one wait
          float v[64];
          tmem_ld32x2(tmem_base + (uint32_t(q * 32) << 16) + uint32_t(buf * TCH + cp * 64), v);
#pragma unroll
          for (int u = 0; u < 64; ++u) sq = fmaf(v[u], v[u], sq);
          if (kBF16 && store_mode != 0) {
            // before the first write into a staging region, the bulk group that last read it (one
            // tile earlier) must be done reading: 4 groups per tile (3-D boxes) or 2 (4-D boxes)
            if (store_mode == 1 || (cp & 1) == 0) {
              if (lane == 0) {
                if (store_mode == 1) bulk_wait_group_read3();
                else bulk_wait_group_read1();
              }
              __syncwarp();
            }
            // row `lane` of box cp (64 channels, 128 bytes), 16-byte chunk u placed with the
            // 128-byte swizzle: chunk index XOR (row % 8)
            const uint32_t box = stage + uint32_t(cp) * (32u * 128u) + uint32_t(lane) * 128u;
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              const uint32_t a = box + ((uint32_t(u) ^ uint32_t(lane & 7)) * 16u);
              asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(a),
                           "r"(pack_bf16x2(v[8 * u], v[8 * u + 1])), "r"(pack_bf16x2(v[8 * u + 2], v[8 * u + 3])),
                           "r"(pack_bf16x2(v[8 * u + 4], v[8 * u + 5])), "r"(pack_bf16x2(v[8 * u + 6], v[8 * u + 7]))
                           : "memory");
            }
            fence_proxy_async_smem();  // box rows visible to the TMA unit
            __syncwarp();
            if (lane == 0) {
              const int rows0 = int(n0) + q * 32;
              if (store_mode == 1) {
                if (rows0 < nend && j0 + 64 * cp < g.d && LOCA_REQUIRE(rows0 >= 0 && (j0 + 64 * cp) % 8 == 0))
                  tma_store_3d(&tmT, stage + uint32_t(cp) * (32u * 128u), int(j0) + 64 * cp, rows0, l);
                bulk_commit_group();
              } else if (cp & 1) {
                const int h = cp >> 1;  // boxes 2h, 2h+1 leave as one 4-D box of two channel blocks
                if (rows0 < nend && j0 + 128 * h < g.d && LOCA_REQUIRE(rows0 >= 0 && j0 % 64 == 0))
                  tma_store_4d(&tmT, stage + uint32_t(h) * (64u * 128u), 0, rows0, int(j0 / 64) + 2 * h, l);
                bulk_commit_group();
              }
            }
            continue;
          }
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const float* vv = v + 32 * hh;
            const int64_t jb = j0 + cp * 64 + hh * 32;
            if (!nv || jb >= g.d) continue;
            if (!LOCA_CHECK_SPAN(rbase + jb, jb + 32 <= g.d ? 32 : g.d - jb, int64_t(g.L) * g.N * g.d)) continue;
            const bool whole = (jb + 32 <= g.d) && (g.d % 8 == 0);
            if (whole) {
              if (kBF16) {
                uint4* o = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(Tout) + rbase + jb);
#pragma unroll
                for (int u = 0; u < 4; ++u)
                  o[u] = make_uint4(pack_bf16x2(vv[8 * u], vv[8 * u + 1]), pack_bf16x2(vv[8 * u + 2], vv[8 * u + 3]),
                                    pack_bf16x2(vv[8 * u + 4], vv[8 * u + 5]), pack_bf16x2(vv[8 * u + 6], vv[8 * u + 7]));
              } else {
                float4* o = reinterpret_cast<float4*>(static_cast<float*>(Tout) + rbase + jb);
#pragma unroll
                for (int u = 0; u < 8; ++u) o[u] = make_float4(vv[4 * u], vv[4 * u + 1], vv[4 * u + 2], vv[4 * u + 3]);
              }
            } else {
#pragma unroll
              for (int u = 0; u < 32; ++u) {
                if (jb + u >= g.d) break;
                if (kBF16)
                  static_cast<__nv_bfloat16*>(Tout)[rbase + jb + u] = __float2bfloat16_rn(vv[u]);
                else
                  static_cast<float*>(Tout)[rbase + jb + u] = vv[u];
              }
            }
          }
        }
        fence_before();
        mbar_arrive(acc_empty(buf));
        sqd += double(sq);
        sq = 0.f;
      }
      if (!ok) break;
      if (partials != nullptr) {
        // one partial per (item, epilogue warp): no synchronisation across warps
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sqd += __shfl_xor_sync(0xffffffffu, sqd, off);
        if (lane == 0 && LOCA_CHECK(((int64_t(l) * g.nd + jt) * g.nchunks + ck) * 4 + q, int64_t(g.L) * g.nd * g.nchunks * 4))
          partials[((int64_t(l) * g.nd + jt) * g.nchunks + ck) * 4 + q] = sqd;
      }
    }
  }

  if (kBF16 && store_mode != 0 && warp >= 4 && warp < 8 && lane == 0) bulk_wait_group0();
  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 8) tmem_dealloc(tmem_base, TMEM_COLS);
}

// out[l] = sum of partials[l * nparts : (l + 1) * nparts] in a fixed order.
__global__ void __launch_bounds__(256) k_reduce_partials(const double* __restrict__ partials,
                                                         int64_t nparts, double* __restrict__ out) {
  __shared__ double sm[256];
  const int l = blockIdx.x;
  double a = 0.0;
  for (int64_t i = threadIdx.x; i < nparts; i += 256)
    if (LOCA_CHECK(int64_t(l) * nparts + i, int64_t(gridDim.x) * nparts)) a += partials[int64_t(l) * nparts + i];
  sm[threadIdx.x] = a;
  __syncthreads();
  for (int w = 128; w > 0; w >>= 1) {
    if (threadIdx.x < w) sm[threadIdx.x] += sm[threadIdx.x + w];
    __syncthreads();
  }
  if (threadIdx.x == 0) out[l] = sm[0];
}

}  // namespace

int64_t targets_num_partials(int64_t N, int64_t d) {
  return ((d + TCH - 1) / TCH) * ((N + CHUNK - 1) / CHUNK) * 4;
}

size_t targets_workspace_bytes(int64_t N, int L, int64_t d) {
  return align256(sizeof(double) * size_t(L) * size_t(targets_num_partials(N, d))) + 256;
}

int targets_max_C() { return kMaxC; }
int targets_max_r() { return kMaxRP; }

cudaError_t launch_targets(const float* E, int64_t N, int C, const float* P, const float* Q,
                           int L, int r, int64_t d, void* T, int t_dtype, double* tsq,
                           void* workspace, int32_t* status, cudaStream_t s) {
  if (N == 0 || d == 0) {
    if (tsq) return cudaMemsetAsync(tsq, 0, sizeof(double) * L, s);
    return cudaSuccess;
  }
  Geo g;
  g.N = N;
  g.d = d;
  g.C = C;
  g.r = r;
  g.rp = (r + 7) / 8 * 8;
  g.L = L;
  g.nd = (d + TCH - 1) / TCH;
  g.nchunks = (N + CHUNK - 1) / CHUNK;
  g.items = int64_t(L) * g.nd * g.nchunks;
  double* partials = tsq ? static_cast<double*>(workspace) : nullptr;
  int32_t* abort_flag = reinterpret_cast<int32_t*>(
      static_cast<char*>(workspace) + align256(sizeof(double) * size_t(L) * size_t(targets_num_partials(N, d))));
  cudaError_t e = cudaMemsetAsync(abort_flag, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  int64_t grid = sm_count();
  if (grid > g.items) grid = g.items;
  // bf16 output with 16-byte rows: tiles leave through TMA stores, 128-byte swizzled boxes of 64
  // channels x 32 tokens.  d % 64 == 0: a 4-D view (64 channels, token, channel block, block) and
  // boxes of two channel blocks (store_mode 2); else a 3-D view (channel, token, block), one box per
  // 64 channels (store_mode 1).  Otherwise plain stores (store_mode 0).
  CUtensorMap tmT;
  memset(&tmT, 0, sizeof(tmT));
  int store_mode = 0;
  if (t_dtype == LOCA_BF16 && d % 8 == 0 && N < (int64_t(1) << 31) && d < (int64_t(1) << 31)) {
    auto fn = tensor_map_encoder();
    if (fn != nullptr && d % 64 == 0) {
      cuuint64_t dims[4] = {64, cuuint64_t(N), cuuint64_t(d / 64), cuuint64_t(L)};
      cuuint64_t strides[3] = {cuuint64_t(d) * 2, 128, cuuint64_t(N) * cuuint64_t(d) * 2};
      cuuint32_t box[4] = {64, 32, 2, 1};
      cuuint32_t estr[4] = {1, 1, 1, 1};
      if (fn(&tmT, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, T, dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS)
        store_mode = 2;
    }
    if (fn != nullptr && store_mode == 0) {
      cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(N), cuuint64_t(L)};
      cuuint64_t strides[2] = {cuuint64_t(d) * 2, cuuint64_t(N) * cuuint64_t(d) * 2};
      cuuint32_t box[3] = {64, 32, 1};
      cuuint32_t estr[3] = {1, 1, 1};
      if (fn(&tmT, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, T, dims, strides, box, estr,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS)
        store_mode = 1;
    }
  }
  const Layout lay = layout_for(g.rp);
  const size_t shm = lay.total;
  const unsigned long long limit = wait_limit_ns();
  if (t_dtype == LOCA_BF16) {
    e = cudaFuncSetAttribute(k_targets_tc<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets_tc<true><<<unsigned(grid), NTHREADS, shm, s>>>(E, P, Q, g, T, tmT, store_mode, partials, status,
                                                             abort_flag, limit);
  } else {
    e = cudaFuncSetAttribute(k_targets_tc<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
    if (e != cudaSuccess) return e;
    k_targets_tc<false><<<unsigned(grid), NTHREADS, shm, s>>>(E, P, Q, g, T, tmT, 0, partials, status,
                                                              abort_flag, limit);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess || tsq == nullptr) return e;
  k_reduce_partials<<<L, 256, 0, s>>>(partials, targets_num_partials(N, d), tsq);
  return cudaGetLastError();
}

}  // namespace loca
