// Gram and cross-product statistics on the sm_103a tensor cores (Eq. 9; S7):
//   Gram_l  (+)= X_l^T X_l          Cross_l (+)= alpha_l T_l^T X_l        (d x d, fp32)
// with X_l, T_l token-major bf16 (N x d) and the token axis as the reduction axis.
//
// Design (one persistent CTA per SM, 192 threads):
//   warp 0       TMA producer: 3-D tensor maps over (channel, token, block) with 128-byte
//                swizzle; boxes of 64 channels x 64 tokens land as the MN-major canonical
//                layout the tensor core reads (channels contiguous, one 128-byte row per token).
//   warp 1       owns 512 TMEM columns and issues tcgen05.mma (kind::f16, bf16 x bf16 -> fp32,
//                M = 128, N = 256, K = 16, both operands MN-major) from one thread.
//   warps 2-5    epilogue: tcgen05.ld of the two 128 x 256 fp32 accumulators, scale, store.
// Work item = one 256-channel column tile nt of X (the B operand, loaded once per stage) and up
// to two 128-row accumulators that share it: Gram tiles that touch the upper triangle and all
// cross tiles of that column, paired in order.  Sharing B gives 128 flop per byte of operand
// traffic.  Gram elements (i, j) with i <= j are stored directly and mirrored to (j, i), so each
// output element is written by exactly one thread (deterministic, no atomics).
// Pipeline: 3 stages of 64 tokens (64 KB each); stage release and accumulator hand-off through
// tcgen05.commit -> mbarrier.  Every wait is bounded: on expiry the CTA records
// LOCA_ERR_TIMEOUT in the status word, sets a launch-local abort flag that makes every other
// wait give up, drains its own copies and MMAs, frees TMEM and returns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>

#include <mutex>

#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

constexpr int BM = 128;                           // accumulator rows (channels of X or T)
constexpr int BN = 256;                           // accumulator columns (channels of X)
constexpr int BK = 64;                            // tokens per pipeline stage
constexpr int STAGES = 3;
constexpr int SUB_BYTES = 64 * BK * 2;            // one TMA box: 64 channels x 64 tokens (8 KB)
constexpr int A_BYTES = BM * BK * 2;              // 16 KB
constexpr int B_BYTES = BN * BK * 2;              // 32 KB
constexpr int STAGE_BYTES = 2 * A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 512;
constexpr int NUM_THREADS = 192;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /* align slack */ + 256 /* barriers */;

// Instruction descriptor (kind::f16): D fp32, A bf16, B bf16, A and B MN-major, N, M.
constexpr uint32_t IDESC = tc::idesc(1, 1, 1, 1, BM, BN);

using namespace tc;

// ------------------------------------------------------------------ work items
struct Geo {
  int L, d, N;
  int nM, nN;       // row tiles (128) and column tiles (256)
  int per_block;    // work items per block l
};

// Gram row tiles of column tile nt that contain an element with row <= column.
__device__ __host__ __forceinline__ int gram_rows(const Geo& g, int nt) {
  int last = nt * BN + BN - 1;
  if (last > g.d - 1) last = g.d - 1;
  int c = last / BM + 1;
  return c < g.nM ? c : g.nM;
}
__device__ __host__ __forceinline__ int items_of_col(const Geo& g, int nt) {
  return (gram_rows(g, nt) + g.nM + 1) / 2;
}

struct Item {
  int l, nt;
  int nslots;
  int kind[2];  // 0 = Gram (rows from X), 1 = cross (rows from T)
  int mt[2];
};

__device__ __forceinline__ Item decode(const Geo& g, int it) {
  Item r;
  r.l = it / g.per_block;
  int rem = it - r.l * g.per_block;
  int nt = 0;
  for (;; ++nt) {
    const int c = items_of_col(g, nt);
    if (rem < c) break;
    rem -= c;
  }
  r.nt = nt;
  const int ng = gram_rows(g, nt);
  const int len = ng + g.nM;
  r.nslots = 0;
  for (int q = 2 * rem; q < 2 * rem + 2 && q < len; ++q) {
    r.kind[r.nslots] = q < ng ? 0 : 1;
    r.mt[r.nslots] = q < ng ? q : q - ng;
    ++r.nslots;
  }
  return r;
}

// ------------------------------------------------------------------ kernel
__global__ void __launch_bounds__(NUM_THREADS, 1)
    k_gram_cross_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmT,
                    Geo g, int total_items, const float* __restrict__ alpha, int zero_first,
                    float* __restrict__ gram, float* __restrict__ cross, int32_t* status,
                    int32_t* abort_flag, unsigned long long limit_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
  // bars[0..S-1] full, [S..2S-1] empty, [2S] acc_full, [2S+1] acc_empty, [2S+2] drain
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * STAGES + 4);
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (STAGES + s); };
  const uint32_t acc_full = bar_base + 8u * (2 * STAGES);
  const uint32_t acc_empty = bar_base + 8u * (2 * STAGES + 1);
  const uint32_t drain_bar = bar_base + 8u * (2 * STAGES + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const WaitCtl wc{status, abort_flag, limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 128);
    mbar_init(drain_bar, 1);
    mbar_init_fence();
    prefetch_tensormap(&tmX);
    prefetch_tensormap(&tmT);
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), TMEM_COLS);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int nkb = (g.N + BK - 1) / BK;

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer
      int stage = 0;
      uint32_t phase = 0;
      uint32_t pending = 0, pending_par = 0;  // stages with loads in flight, their phase parity
      bool ok = true;
      for (int it = blockIdx.x; it < total_items && ok; it += gridDim.x) {
        const Item w = decode(g, it);
        const uint32_t bytes = uint32_t(w.nslots) * A_BYTES + B_BYTES;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(empty_bar(stage), phase ^ 1u, wc)) { ok = false; break; }
          const uint32_t fb = full_bar(stage);
          mbar_arrive_expect_tx(fb, bytes);
          const uint32_t st = smem_base + uint32_t(stage) * STAGE_BYTES;
          const int tok = kb * BK;
          for (int s = 0; s < w.nslots; ++s) {
            const CUtensorMap* map = w.kind[s] == 0 ? &tmX : &tmT;
            const uint32_t dst = st + uint32_t(s) * A_BYTES;
            tma_load_3d(dst, map, fb, w.mt[s] * BM, tok, w.l);
            tma_load_3d(dst + SUB_BYTES, map, fb, w.mt[s] * BM + 64, tok, w.l);
          }
          const uint32_t bdst = st + 2u * A_BYTES;
#pragma unroll
          for (int h = 0; h < BN / 64; ++h)
            tma_load_3d(bdst + uint32_t(h) * SUB_BYTES, &tmX, fb, w.nt * BN + h * 64, tok, w.l);
          pending |= 1u << stage;
          pending_par = (pending_par & ~(1u << stage)) | (phase << stage);
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
      }
      if (!ok) {
        // let the copies already issued land before the CTA can exit
        const uint64_t t0 = globaltimer();
        for (int s = 0; s < STAGES; ++s) {
          if (!(pending & (1u << s))) continue;
          while (!mbar_try_wait(full_bar(s), (pending_par >> s) & 1u)) {
            if (globaltimer() - t0 > limit_ns) break;
          }
        }
      }
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {
      // ---------------- MMA issuer
      int stage = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      bool issued = false;
      for (int it = blockIdx.x; it < total_items && ok; it += gridDim.x) {
        const Item w = decode(g, it);
        if (!mbar_wait(acc_empty, acc_phase ^ 1u, wc)) { ok = false; break; }
        fence_after();
        for (int kb = 0; kb < nkb; ++kb) {
          if (!mbar_wait(full_bar(stage), phase, wc)) { ok = false; break; }
          fence_after();
          const uint32_t st = smem_base + uint32_t(stage) * STAGE_BYTES;
          const uint32_t bsm = st + 2u * A_BYTES;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint64_t bd = sdesc(bsm + uint32_t(kk) * 2048u, SUB_BYTES, 1024u, kSwizzle128B);
            for (int s = 0; s < w.nslots; ++s) {
              const uint64_t ad = sdesc(st + uint32_t(s) * A_BYTES + uint32_t(kk) * 2048u,
                                        SUB_BYTES, 1024u, kSwizzle128B);
              mma_f16(tmem_base + uint32_t(s) * BN, ad, bd, IDESC, (kb | kk) != 0 ? 1u : 0u);
            }
          }
          issued = true;
          mma_commit(empty_bar(stage));  // frees the stage once these MMAs have read it
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        mma_commit(acc_full);  // accumulators complete
        acc_phase ^= 1u;
      }
      if (!ok && issued) {
        mma_commit(drain_bar);
        const uint64_t t0 = globaltimer();
        while (!mbar_try_wait(drain_bar, 0)) {
          if (globaltimer() - t0 > limit_ns) break;
        }
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 2..5, TMEM lane quarter = warp % 4
    const int q = warp & 3;
    const int row_in_tile = q * 32 + lane;
    uint32_t acc_phase = 0;
    for (int it = blockIdx.x; it < total_items; it += gridDim.x) {
      const Item w = decode(g, it);
      const bool ok = mbar_wait(acc_full, acc_phase, wc);
      if (!__all_sync(0xffffffffu, ok)) break;  // warp-uniform decision, warp reconverged
      fence_after();
      const float al = alpha[w.l];
      for (int s = 0; s < w.nslots; ++s) {
        const bool is_gram = w.kind[s] == 0;
        float* out = (is_gram ? gram : cross) + int64_t(w.l) * g.d * g.d;
        const int i = w.mt[s] * BM + row_in_tile;
        const float sc = is_gram ? 1.f : al;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
          float v[32];
          tmem_ld32(tmem_base + (uint32_t(q * 32) << 16) + uint32_t(s * BN + c * 32), v);
          const int j0 = w.nt * BN + c * 32;
          if (i >= g.d || j0 >= g.d) continue;
          float* orow = out + int64_t(i) * g.d;
          const bool whole = (j0 + 32 <= g.d) && (!is_gram || i <= j0);
          if (whole) {
            float4* p = reinterpret_cast<float4*>(orow + j0);
#pragma unroll
            for (int u = 0; u < 8; ++u) {
              float4 x = make_float4(sc * v[4 * u], sc * v[4 * u + 1], sc * v[4 * u + 2],
                                     sc * v[4 * u + 3]);
              if (!zero_first) {
                const float4 o = p[u];
                x.x += o.x; x.y += o.y; x.z += o.z; x.w += o.w;
              }
              p[u] = x;
            }
          } else {
#pragma unroll
            for (int u = 0; u < 32; ++u) {
              const int j = j0 + u;
              if (j >= g.d) break;
              if (is_gram && i > j) continue;
              const float x = sc * v[u];
              orow[j] = zero_first ? x : orow[j] + x;
            }
          }
          if (is_gram) {
            // mirror (i, j), i < j, to (j, i): for fixed j the warp writes 32 consecutive i
#pragma unroll 4
            for (int u = 0; u < 32; ++u) {
              const int j = j0 + u;
              if (j >= g.d) break;
              if (i < j) {
                float* p = out + int64_t(j) * g.d + i;
                *p = zero_first ? v[u] : *p + v[u];
              }
            }
          }
        }
      }
      fence_before();
      mbar_arrive(acc_empty);
      acc_phase ^= 1u;
    }
  }

  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, TMEM_COLS);
}

// ------------------------------------------------------------------ host side
bool make_map(CUtensorMap* m, const void* base, int L, int64_t N, int64_t d) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(N), cuuint64_t(L)};
  cuuint64_t strides[2] = {cuuint64_t(d) * 2, cuuint64_t(N) * cuuint64_t(d) * 2};
  cuuint32_t box[3] = {64, BK, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  const CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                        strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                        CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_gram_cross_tc(const void* X, const void* T, int L, int64_t N, int64_t d,
                                 const float* alpha, int zero_first, float* gram, float* cross,
                                 int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  CUtensorMap mx, mt;
  if (!make_map(&mx, X, L, N, d) || !make_map(&mt, T, L, N, d)) return cudaErrorInvalidValue;
  Geo g;
  g.L = L;
  g.d = int(d);
  g.N = int(N);
  g.nM = int((d + BM - 1) / BM);
  g.nN = int((d + BN - 1) / BN);
  g.per_block = 0;
  for (int nt = 0; nt < g.nN; ++nt) g.per_block += items_of_col(g, nt);
  const int total = g.per_block * L;
  int grid = sm_count();
  if (grid > total) grid = total;
  cudaError_t e = cudaMemsetAsync(abort_flag, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(k_gram_cross_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES);
  if (e != cudaSuccess) return e;
  k_gram_cross_tc<<<grid, NUM_THREADS, SMEM_BYTES, s>>>(mx, mt, g, total, alpha, zero_first, gram,
                                                        cross, status, abort_flag,
                                                        4000000000ull /* 4 s per wait */);
  return cudaGetLastError();
}

}  // namespace loca
