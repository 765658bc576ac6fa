// Gram and cross-product statistics on the sm_103a tensor cores (Eq. 9; S7):
//   Gram_l  (+)= X_l^T X_l          Cross_l (+)= alpha_l T_l^T X_l        (d x d, fp32)
// with X_l, T_l token-major bf16 (N x d) and the token axis as the reduction axis.
//
// Design: persistent CTA pairs (clusters of 2, one CTA per SM), 192 threads per CTA.
//   The pair computes 256-row x 256-column accumulator tiles with tcgen05.mma.cta_group::2
//   (kind::f16, bf16 x bf16 -> fp32, M = 256, N = 256, K = 16, both operands MN-major): each CTA
//   loads its own 128 rows of A and its own 128 columns of B, and its TMEM holds its 128 rows of
//   the result.  Per SM a pipeline stage is then 48 KB (two A tiles and half a B tile, 64 tokens)
//   for the MMA work a single-CTA 128 x 256 tile pair needs 64 KB for, so four stages fit in
//   shared memory; the extra stage covers the load latency of 152 SMs streaming the same rows.
//   warp 0       TMA producer (both CTAs): one 4-D load per operand (64-channel blocks of a
//                (64 channels, token, channel block, block) view, 128-byte swizzle) when
//                d % 64 == 0, else one 3-D load per 64-channel block.  The loads of both CTAs
//                count their bytes on the even CTA's full barrier (pair form of the TMA load);
//                the even CTA arms it with the bytes of both.
//   warp 1       owns 512 TMEM columns (two 128 x 256 fp32 accumulators per CTA); in the even
//                CTA one thread issues the MMAs.  Its loop is kept short (descriptors built once,
//                advanced by integer adds; bounded wait entered only if an inline try_wait fails)
//                so that issue keeps pace with the tensor core.
//   warps 2-5    epilogue (both CTAs): tcgen05.ld, scale, stage 32 x 32 boxes in shared memory
//                (128-byte swizzle) and hand them to the TMA unit: a bulk store for the first
//                segment of a zero_first launch, a bulk reduce-add into the fp32 output otherwise.
// Work item = one 256-column tile of X (B) and up to two 256-row accumulators sharing it (Gram
// tiles that touch the upper triangle and all cross tiles of that column, paired in order).
// Segments: an item's token axis is cut into segments of kSegTokens tokens; the accumulators start
// from zero in every segment and each segment's sums are added into the fp32 output.  The tensor
// cores' fp32 accumulation loses a fraction of an ulp of the running sum at every MMA step, always
// toward zero; bounding the steps per accumulator bounds that bias (the output's own additions
// round to nearest).  The MMA issuer waits for the epilogue only until the TMEM reads are done:
// the stores and additions are the TMA unit's.  Each output element has one issuing thread, which
// waits for its previous segment's additions to complete before issuing the next, so the order
// of additions is fixed (deterministic, no atomics).  Gram tiles are written whole; the elements
// below the diagonal are then overwritten with their mirror images by k_gram_mirror, so the Gram
// matrix is exactly symmetric.
// Lockstep: all clusters stream the same token window of X_l and T_l at the same time, so an
// operand line read from HBM is then served from L2 to the other tiles that need it.  The even
// CTA's producer passes a sync point at the start of every work item and every kSyncEvery
// k-blocks within it: it counts the point on a launch-local counter and waits (bounded, as a hint
// only) until every cluster with an item in this round has counted it too.  Without the item-level
// points the clusters drift apart over a few items (items differ in length and epilogue cost), the
// L2 no longer holds what the others read, and the load latency, not the tensor core, sets the
// pace (about 1.25x slower at 7B size); the points within items keep the clusters' token windows
// within ~L2 of each other (HBM re-reads 4.0x -> 2.6x of X and T, 3-4% faster under the power cap).
// Rounds are aligned to blocks: the items are ordered so that a round holds the items of one block
// only, each block filling whole rounds, and the few items left of every block follow at the end;
// a round then streams one block's tiles instead of parts of two.
// Every mbarrier wait is bounded: on expiry the status word gets LOCA_ERR_TIMEOUT, a launch-local
// flag makes every other wait give up, and the roles stop, each CTA's producer at its own point.
// At the end both CTAs meet at a cluster barrier (the odd CTA has posted how many pipeline
// iterations it issued); then the even CTA reconciles its full barriers with what each CTA issued
// (arming what only the odd CTA issued, settling with mbarrier.complete_tx the bytes the odd CTA
// never issued) and waits for every copy to land; the MMAs in flight are waited for and the
// epilogue's bulk copies have completed; only then do both CTAs pass the final cluster barrier
// and free TMEM.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstring>

#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

using namespace tc;

constexpr int BMP = 256;                            // accumulator rows per CTA pair
constexpr int BMC = 128;                            // accumulator rows per CTA (TMEM lanes)
constexpr int BN = 256;                             // accumulator columns (channels of X)
constexpr int BNC = 128;                            // B columns loaded per CTA
constexpr int BK = 64;                              // tokens per pipeline stage
constexpr int STAGES = 4;
constexpr int kSyncEvery = 64;                     // k-blocks between lockstep sync points
constexpr int SUB_BYTES = 64 * BK * 2;              // one 64-channel x 64-token swizzled tile (8 KB)
constexpr int A_BYTES = BMC * BK * 2;               // 16 KB
constexpr int B_BYTES = BNC * BK * 2;               // 16 KB
constexpr int STAGE_BYTES = 2 * A_BYTES + B_BYTES;  // 48 KB
constexpr int TMEM_COLS = 512;
constexpr int kSegTokens = 16384;                   // tokens per accumulation segment
constexpr int EPI_BOX_BYTES = 32 * 32 * 4;          // one 32-row x 32-column fp32 output box
static_assert(kSegTokens % (BK * kSyncEvery) == 0, "segments end on lockstep sync points");

// Instruction descriptor (kind::f16): D fp32, A bf16, B bf16, A and B MN-major, M = 256, N = 256.
constexpr uint32_t IDESC_PAIR = tc::idesc(1, 1, 1, 1, BMP, BN);

// ------------------------------------------------------------------ work items
struct Geo {
  int L, d, N;
  int nM, nN;       // 256-row tiles and 256-column tiles
  int per_block;    // work items per block l
  int full;         // items of each block that fill whole rounds of their own (0: plain order)
  int fused;        // 1: cross items generate their T tile (one accumulator each)
};

// Gram row tiles of column tile nt that contain an element with row <= column.
__device__ __host__ __forceinline__ int gram_rows(const Geo& g, int nt) {
  int last = nt * BN + BN - 1;
  if (last > g.d - 1) last = g.d - 1;
  int c = last / BMP + 1;
  return c < g.nM ? c : g.nM;
}
// Items of column tile nt: the Gram row tiles and the cross row tiles paired in order, or, with
// fused targets, Gram tiles paired and every cross tile an item of its own.
__device__ __host__ __forceinline__ int items_of_col(const Geo& g, int nt) {
  return g.fused ? (gram_rows(g, nt) + 1) / 2 + g.nM : (gram_rows(g, nt) + g.nM + 1) / 2;
}

struct Item {
  int l, nt;
  int nslots;
  int kind[2];  // 0 = Gram (rows from X), 1 = cross (rows from T)
  int mt[2];    // 256-row tile index
};

// Round-aligned order: a round is the items cid + round * (clusters).  The first `full` items of
// block l (a multiple of the cluster count) fill rounds of block l alone, so a round streams the
// tiles of one block; the per_block - full items left of every block come after all blocks.
__device__ __forceinline__ Item decode(const Geo& g, int it) {
  Item r;
  int rem;
  if (g.full > 0 && it < g.L * g.full) {
    r.l = it / g.full;
    rem = it - r.l * g.full;
  } else if (g.full > 0) {
    const int q = g.per_block - g.full;  // > 0 here: it < L * per_block
    const int j = it - g.L * g.full;
    r.l = j / q;
    rem = g.full + (j - r.l * q);
  } else {
    r.l = it / g.per_block;
    rem = it - r.l * g.per_block;
  }
  int nt = 0;
  for (;; ++nt) {
    const int c = items_of_col(g, nt);
    if (rem < c) break;
    rem -= c;
  }
  r.nt = nt;
  const int ng = gram_rows(g, nt);
  r.nslots = 0;
  if (g.fused && rem >= (ng + 1) / 2) {  // a cross tile whose T tile the kernel generates
    r.kind[0] = 1;
    r.mt[0] = rem - (ng + 1) / 2;
    r.nslots = 1;
    return r;
  }
  const int len = g.fused ? ng : ng + g.nM;
  for (int q = 2 * rem; q < 2 * rem + 2 && q < len; ++q) {
    r.kind[r.nslots] = q < ng ? 0 : 1;
    r.mt[r.nslots] = q < ng ? q : q - ng;
    ++r.nslots;
  }
  return r;
}

// ------------------------------------------------------------------ fused targets
// With fused targets a cross item's A operand, the T tile (256 channels x 64 tokens per stage),
// is generated inside the kernel from U = E P_l (tokens x r) and Q_l (r x channels):
//   k_fused_u            before the kernel: U_l = E P_l for every block (fp32, the same chain as
//                        k_targets_tc) as bf16 hi / lo parts, N x rp each, in the workspace;
//   warp 6 (both CTAs)   writes, per cross item, Q_l^T for the CTA's 128 channels as bf16 hi / lo
//                        parts (K-major), and per stage copies U for the CTA's 32 tokens of the
//                        stage (K-major, the next stage's rows already in registers) into the
//                        stage's second A region, which cross items do not load;
//   warp 7 (even CTA)    D = Q^T U on the tensor cores as Qh Uh + Qh Ul + Ql Uh (pair MMA,
//                        M = 256 channels, N = 64 tokens, K = 16), into one of four 64-column TMEM
//                        buffers beside the accumulator, as far ahead as the buffers allow; a
//                        thread of its own, so that its commits wait only for its own MMAs;
//   warps 2-5, 8-11      read D (fp32, one channel per lane; warps 2-5 the first 32 tokens,
//                        8-11 the other 32), round it to bf16 once and write it, channel pairs
//                        packed in 32-bit words, into the stage's first A region in the layout
//                        the TMA load of T would have produced (64-channel x 64-token boxes,
//                        128-byte swizzle); the MMA thread waits for all of them.
// The split keeps ~2^-17 of each product, so T is rounded to bf16 from a near-fp32 value, as in
// k_targets_tc.  Cross items take one accumulator (256 TMEM columns) so that the T buffers fit.
struct Fuse {
  const __nv_bfloat16* Uh;  // L x N x rp: bf16 hi part of U_l = E P_l (zero beyond r)
  const __nv_bfloat16* Ul;  // L x N x rp: bf16 lo part, U_l - hi
  const float* Q;           // L x r x d
  int r, rp;                // rp: r padded to 16 or 32
};
constexpr int U_ROWS = BK / 2;  // tokens of a stage per CTA (the pair MMA's N = 64 split in two)
constexpr uint32_t IDESC_TGEN = tc::idesc(1, 1, 0, 0, BMP, BK);  // bf16, K-major, M = 256, N = 64
constexpr uint32_t TGEN_COL = BN;  // TMEM column of the first T buffer (after one accumulator)
constexpr int TGEN_BUFS = 4;       // 64-column T buffers: the other half of TMEM

// K-major, no-swizzle canonical bf16 tile with rp columns: 8-row x 8-element core matrices,
// K-adjacent ones 128 bytes apart, 8-row groups rp * 16 bytes apart
__device__ __forceinline__ uint32_t kmaj16_off(int m, int s, int rp) {
  return uint32_t(m >> 3) * uint32_t(rp * 16) + uint32_t(s >> 3) * 128u + uint32_t(m & 7) * 16u +
         uint32_t(s & 7) * 2u;
}
// MN-major 128-byte swizzled A tile of 128 channels x 64 tokens (two 64-channel boxes)
__device__ __forceinline__ uint32_t mnmaj_off(int c, int t) {
  return uint32_t(c >> 6) * uint32_t(SUB_BYTES) + uint32_t(t) * 128u +
         ((uint32_t((c & 63) >> 3) ^ uint32_t(t & 7)) << 4) + uint32_t(c & 7) * 2u;
}
__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16& hi, __nv_bfloat16& lo) {
  hi = __float2bfloat16_rn(x);
  lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

// U_l = E P_l for every block as bf16 hi / lo parts (one thread per token; the fp32 chain over the C
// label columns of the targets kernel), rows of rp values, zero beyond r.
__global__ void __launch_bounds__(256) k_fused_u(const float* __restrict__ E, int64_t N, int C,
                                                 const float* __restrict__ P, int r, int rp,
                                                 __nv_bfloat16* __restrict__ Uh, __nv_bfloat16* __restrict__ Ul) {
  const int l = blockIdx.y;
  const int64_t n = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
  if (n >= N) return;
  if (!LOCA_CHECK_SPAN(n * C, C, N * C) || !LOCA_CHECK_SPAN((int64_t(l) * N + n) * rp, rp, int64_t(gridDim.y) * N * rp))
    return;
  const float* Pl = P + int64_t(l) * C * r;
  float u[32];
#pragma unroll
  for (int s = 0; s < 32; ++s) u[s] = 0.f;
  const float* er = E + n * C;
  for (int c = 0; c < C; ++c) {
    const float ec = er[c];
    const float* pr = Pl + c * r;
#pragma unroll
    for (int s = 0; s < 32; ++s)
      if (s < r) u[s] = fmaf(ec, __ldg(pr + s), u[s]);
  }
  __nv_bfloat16* hrow = Uh + (int64_t(l) * N + n) * rp;
  __nv_bfloat16* lrow = Ul + (int64_t(l) * N + n) * rp;
#pragma unroll
  for (int s = 0; s < 32; ++s) {
    if (s < rp) {
      __nv_bfloat16 h, lo;
      split_bf16(u[s], h, lo);
      hrow[s] = h;
      lrow[s] = lo;
    }
  }
}

template <bool kFused>
struct Cfg {
  static constexpr int kThreads = kFused ? 384 : 192;
  static constexpr int kBufs = kFused ? 1 : 2;  // staging boxes per epilogue warp
  static constexpr int kEpiBytes = 4 * kBufs * EPI_BOX_BYTES;
  static constexpr int kQBytes = kFused ? 16384 : 0;  // Q^T hi / lo, 128 channels x 32
  // full[S], empty[S], acc_full, acc_empty, drain; fused: u_full[S], a_ready[S], tgen_full[TB],
  // tgen_empty[TB], q_full, q_free, u_go[S], u_free[S], tg_go, tg_drain
  static constexpr int kBars = kFused ? 6 * STAGES + 7 + 2 * TGEN_BUFS : 2 * STAGES + 3;
  static constexpr int kBarBytes = kFused ? 512 : 256;
  static constexpr int kSmem = STAGES * STAGE_BYTES + kEpiBytes + kQBytes + 1024 + kBarBytes;
};
static_assert(Cfg<false>::kSmem <= 232448 && Cfg<true>::kSmem <= 232448, "shared memory per CTA");
static_assert(Cfg<true>::kBars * 8 + 8 <= Cfg<true>::kBarBytes, "barrier area");  // + TMEM slot, odd count

// ------------------------------------------------------------------ kernel
template <bool kFused>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(Cfg<kFused>::kThreads, 1)
    k_gram_cross_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmT,
                    const __grid_constant__ CUtensorMap tmXa, const __grid_constant__ CUtensorMap tmTa,
                    const __grid_constant__ CUtensorMap tmXb, const __grid_constant__ CUtensorMap tmG,
                    const __grid_constant__ CUtensorMap tmC, int blocked, Geo g, int total_items, int seg_kb,
                    const float* __restrict__ alpha, int zero_first, int32_t* status, int32_t* abort_flag,
                    uint32_t* round_ctr, unsigned long long limit_ns, unsigned long long sync_ns, Fuse fz) {
  using K = Cfg<kFused>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* epi = smem + STAGES * STAGE_BYTES;  // 1024-aligned: the boxes use the 128-byte swizzle
  uint8_t* qbuf = epi + K::kEpiBytes;          // fused: Q^T hi at +0, lo at +8 KB
  uint64_t* bars = reinterpret_cast<uint64_t*>(qbuf + K::kQBytes);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + K::kBars);
  uint32_t* odd_issued = tmem_slot + 1;  // even CTA: pipeline iterations the odd CTA issued
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (STAGES + s); };
  const uint32_t acc_full = bar_base + 8u * (2 * STAGES);
  const uint32_t acc_empty = bar_base + 8u * (2 * STAGES + 1);
  const uint32_t drain_bar = bar_base + 8u * (2 * STAGES + 2);
  auto u_full = [&](int s) { return bar_base + 8u * (2 * STAGES + 3 + s); };
  auto a_ready = [&](int s) { return bar_base + 8u * (3 * STAGES + 3 + s); };
  auto tgen_full = [&](int b) { return bar_base + 8u * (4 * STAGES + 3 + b); };
  auto tgen_empty = [&](int b) { return bar_base + 8u * (4 * STAGES + 3 + TGEN_BUFS + b); };
  const uint32_t q_full = bar_base + 8u * (4 * STAGES + 3 + 2 * TGEN_BUFS);
  const uint32_t q_free = bar_base + 8u * (4 * STAGES + 4 + 2 * TGEN_BUFS);
  auto u_go = [&](int s) { return bar_base + 8u * (4 * STAGES + 5 + 2 * TGEN_BUFS + s); };
  auto u_free = [&](int s) { return bar_base + 8u * (5 * STAGES + 5 + 2 * TGEN_BUFS + s); };
  const uint32_t tg_go = bar_base + 8u * (6 * STAGES + 5 + 2 * TGEN_BUFS);
  const uint32_t tg_drain = bar_base + 8u * (6 * STAGES + 6 + 2 * TGEN_BUFS);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cid = int(cluster_id_x());
  const int ncl = int(ncluster_x());
  const WaitCtl wc{status, abort_flag, limit_ns};
  // bytes one CTA loads per stage of an item (fused cross items load only X)
  auto item_bytes = [&](const Item& w) -> uint32_t {
    if (kFused && w.kind[0] == 1) return uint32_t(B_BYTES);
    return uint32_t(w.nslots) * A_BYTES + B_BYTES;
  };
  auto fused_cross = [&](const Item& w) { return kFused && w.kind[0] == 1; };


  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 8);  // lane 0 of the 4 epilogue warps of each CTA
    mbar_init(drain_bar, 1);
    if (kFused) {
      for (int s = 0; s < STAGES; ++s) {
        mbar_init(u_full(s), 2);    // lane 0 of warp 6 of each CTA
        mbar_init(a_ready(s), 16);  // lane 0 of the 8 converting warps of each CTA
      }
      for (int b = 0; b < TGEN_BUFS; ++b) {
        mbar_init(tgen_full(b), 1);
        mbar_init(tgen_empty(b), 16);
      }
      mbar_init(tg_go, 1);     // the even CTA's MMA thread: earlier items' statistics complete
      mbar_init(tg_drain, 1);  // the T thread's own MMAs, before TMEM is freed
      mbar_init(q_full, 2);
      mbar_init(q_free, 1);
      for (int s = 0; s < STAGES; ++s) {
        mbar_init(u_go(s), 1);    // this CTA's TMA producer
        mbar_init(u_free(s), 1);  // the T generation that read the stage's U
      }
    }
    *odd_issued = 0;
    mbar_init_fence();
    if (blocked) {
      prefetch_tensormap(&tmXa);
      prefetch_tensormap(&tmTa);
      prefetch_tensormap(&tmXb);
    } else {
      prefetch_tensormap(&tmX);
      prefetch_tensormap(&tmT);
    }
    prefetch_tensormap(&tmG);
    prefetch_tensormap(&tmC);
  }
  if (warp == 1) tmem_alloc_pair(smem_u32(tmem_slot), TMEM_COLS);
  fence_before();
  cluster_sync();  // barriers of both CTAs initialised, TMEM allocated
  fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int nkb = (g.N + BK - 1) / BK;
  const int nseg = (nkb + seg_kb - 1) / seg_kb;
  // One warp's share of a generated T tile: D rows (channels) of lane quarter q, tokens
  // [t0, t0 + 32), from TMEM buffer tg % TGEN_BUFS -> bf16 -> stage s's A tile, channel pairs packed
  // into 32-bit words (lane pairs trade one value).  False when a wait gave up (warp-uniform).
  auto convert_t = [&](int q, int t0, uint32_t tg, uint32_t j) -> bool {
    const uint32_t b = tg % TGEN_BUFS;
    const bool okw = mbar_wait_cluster(tgen_full(b), (tg / TGEN_BUFS) & 1u, wc);
    if (!__all_sync(0xffffffffu, okw)) return false;
    fence_after();
    float v[32];
    tmem_ld32(tmem_base + (uint32_t(q * 32) << 16) + TGEN_COL + b * uint32_t(BK) + uint32_t(t0), v);
    fence_before();
    __syncwarp();
    if (lane == 0) {
      if (leader) mbar_arrive(tgen_empty(b));
      else mbar_arrive_remote(mapa_shared(tgen_empty(b), 0));
    }
    // the stage's A tile is free once the statistics MMAs of its previous use have completed
    const int s = int(j % STAGES);
    const bool oke = mbar_wait_cluster(empty_bar(s), ((j / STAGES) & 1u) ^ 1u, wc);
    if (!__all_sync(0xffffffffu, oke)) return false;
    uint8_t* at = smem + s * STAGE_BYTES;
    const int c = q * 32 + lane;
    const bool odd = (lane & 1) != 0;
    const int cb = c & ~1;
#pragma unroll
    for (int t = 0; t < 32; t += 2) {
      // even lanes write token t of channels (c, c + 1), odd lanes token t + 1 of (c - 1, c)
      const float recv = __shfl_xor_sync(0xffffffffu, odd ? v[t] : v[t + 1], 1);
      const float lo = odd ? recv : v[t];
      const float hi = odd ? v[t + 1] : recv;
      const __nv_bfloat162 pr = __floats2bfloat162_rn(lo, hi);
      *reinterpret_cast<__nv_bfloat162*>(at + mnmaj_off(cb, t0 + t + (odd ? 1 : 0))) = pr;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      if (leader) mbar_arrive(a_ready(s));
      else mbar_arrive_remote(mapa_shared(a_ready(s), 0));
    }
    return true;
  };
  uint32_t iters_done = 0;  // producer: pipeline iterations this CTA issued

  if (warp == 0) {
    if (lane == 0) {
      // ---------------- TMA producer (both CTAs): this CTA's rows of A and columns of B
      int stage = 0;
      uint32_t phase = 0;
      uint32_t iter = 0;  // pipeline iterations issued by this CTA
      bool ok = true;
      bool sync = leader;  // dropped for the rest of the launch if a wait runs out
      // sync points: each item counts one every kSyncEvery k-blocks and one at its end (P per item)
      const int P = (nkb + kSyncEvery - 1) / kSyncEvery;
      uint32_t before = 0;  // counts expected from all earlier rounds
      auto wait_for = [&](uint32_t target) {  // a hint: bounded, no error
        const uint64_t t0 = globaltimer();
        while (*reinterpret_cast<volatile uint32_t*>(round_ctr) < target) {
          if (globaltimer() - t0 > sync_ns) {
            sync = false;
            break;
          }
        }
      };
      uint32_t round = 0;
      for (int it = cid; it < total_items && ok; it += ncl, ++round) {
        // clusters with an item in this round (the last round may be partial)
        const int left = total_items - int(round) * ncl;
        const uint32_t active = uint32_t(left < ncl ? left : ncl);
        if (sync && round > 0) wait_for(before);  // every cluster finished issuing its last item
        const Item w = decode(g, it);
        const uint32_t bytes_one = item_bytes(w);
        const bool gen = fused_cross(w);
        for (int kb = 0; kb < nkb; ++kb) {
          if (leader && kb > 0 && kb % kSyncEvery == 0) {
            atomicAdd(round_ctr, 1u);
            if (sync) wait_for(before + active * uint32_t(kb / kSyncEvery));
          }
          if (!mbar_try_wait_cluster(empty_bar(stage), phase ^ 1u) &&
              !mbar_wait_cluster(empty_bar(stage), phase ^ 1u, wc)) {
            ok = false;
            break;
          }
          if (leader) mbar_arrive_expect_tx(full_bar(stage), 2u * bytes_one);
          // the stage is free: this CTA's U may be written (later stages of the item: see u_free)
          if (gen && kb < STAGES) mbar_arrive(u_go(stage));
          const uint32_t fb = mapa_shared(full_bar(stage), 0);
          const uint32_t st = smem_base + uint32_t(stage) * STAGE_BYTES;
          const uint32_t bdst = st + 2u * A_BYTES;
          const int tok = kb * BK;
          const int col0 = w.nt * BN + int(rank) * BNC;
          // the stage is armed: a failed check is recorded, the loads (out-of-range boxes are
          // filled by the TMA unit) still run so that the barrier completes
          (void)LOCA_REQUIRE(tok >= 0 && col0 % 64 == 0);
          if (blocked) {
            if (!gen)
              for (int s = 0; s < w.nslots; ++s)
                tma_load_4d_pair(st + uint32_t(s) * A_BYTES, w.kind[s] == 0 ? &tmXa : &tmTa, fb, 0, tok,
                                 (w.mt[s] * BMP + int(rank) * BMC) / 64, w.l);
            tma_load_4d_pair(bdst, &tmXb, fb, 0, tok, col0 / 64, w.l);
          } else {
            if (!gen)
              for (int s = 0; s < w.nslots; ++s) {
                const CUtensorMap* map = w.kind[s] == 0 ? &tmX : &tmT;
                const uint32_t dst = st + uint32_t(s) * A_BYTES;
                const int row0 = w.mt[s] * BMP + int(rank) * BMC;
                (void)LOCA_REQUIRE(row0 % 64 == 0);
                tma_load_3d_pair(dst, map, fb, row0, tok, w.l);
                tma_load_3d_pair(dst + SUB_BYTES, map, fb, row0 + 64, tok, w.l);
              }
            tma_load_3d_pair(bdst, &tmX, fb, col0, tok, w.l);
            tma_load_3d_pair(bdst + SUB_BYTES, &tmX, fb, col0 + 64, tok, w.l);
          }
          ++iter;
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
        }
        if (ok && leader) atomicAdd(round_ctr, 1u);
        before += active * uint32_t(P);
      }
      // the odd CTA posts how many iterations it issued (read by the even CTA after the barrier)
      if (!leader) st_shared_cluster_u32(mapa_shared(smem_u32(odd_issued), 0), iter);
      iters_done = iter;
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ---------------- MMA issuer (even CTA)
      int stage = 0;
      uint32_t phase = 0, acc_phase = 0;
      bool ok = true;
      bool issued = false;
      const uint64_t a_desc0 = sdesc(smem_base, SUB_BYTES, 1024u, kSwizzle128B);
      const uint64_t b_desc0 = sdesc(smem_base + 2u * A_BYTES, SUB_BYTES, 1024u, kSwizzle128B);
      constexpr uint64_t kStageStep = STAGE_BYTES >> 4, kSlotStep = A_BYTES >> 4, kKStep = 2048 >> 4;
      const uint32_t d0 = tmem_base, d1 = tmem_base + uint32_t(BN);
      uint32_t cu[STAGES] = {0, 0, 0, 0};  // fused: cross uses of each stage (a_ready phases)
      for (int it = cid; it < total_items && ok; it += ncl) {
        const Item w = decode(g, it);
        const bool two = w.nslots == 2;
        const bool gen = fused_cross(w);
        if (gen) {
          // the previous item's accumulators (TMEM columns the T buffers reuse) have been read:
          // the T thread may start this item
          if (!mbar_try_wait_cluster(acc_empty, acc_phase ^ 1u) &&
              !mbar_wait_cluster(acc_empty, acc_phase ^ 1u, wc)) {
            ok = false;
            break;
          }
          fence_after();
          mbar_arrive(tg_go);  // both CTAs: the T thread and the converting warps
          mbar_arrive_remote(mapa_shared(tg_go, 1));
        }
        for (int kb = 0; kb < nkb; ++kb) {
          const int in_seg = kb % seg_kb;
          if (in_seg == 0 && !(gen && kb == 0)) {  // a new segment: the epilogue has read the sums
            if (!mbar_try_wait_cluster(acc_empty, acc_phase ^ 1u) &&
                !mbar_wait_cluster(acc_empty, acc_phase ^ 1u, wc)) {
              ok = false;
              break;
            }
            fence_after();
          }
          if (!mbar_try_wait_cluster(full_bar(stage), phase) &&
              !mbar_wait_cluster(full_bar(stage), phase, wc)) {
            ok = false;
            break;
          }
          if (gen) {  // this stage's T tile has been written by both CTAs
            if (!mbar_try_wait_cluster(a_ready(stage), cu[stage] & 1u) &&
                !mbar_wait_cluster(a_ready(stage), cu[stage] & 1u, wc)) {
              ok = false;
              break;
            }
            ++cu[stage];
          }
          fence_after();
          const uint64_t so = uint64_t(stage) * kStageStep;
          const uint64_t ad = a_desc0 + so, bd = b_desc0 + so;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint32_t acc = (in_seg | kk) != 0 ? 1u : 0u;
            mma_f16_pair(d0, ad + kk * kKStep, bd + kk * kKStep, IDESC_PAIR, acc);
            if (two) mma_f16_pair(d1, ad + kSlotStep + kk * kKStep, bd + kk * kKStep, IDESC_PAIR, acc);
          }
          issued = true;
          mma_commit_pair_mc(empty_bar(stage), 0x3);  // frees the stage in both CTAs
          if (++stage == STAGES) { stage = 0; phase ^= 1u; }
          if (in_seg == seg_kb - 1 || kb == nkb - 1) {
            mma_commit_pair_mc(acc_full, 0x3);  // this segment's sums complete in both CTAs
            acc_phase ^= 1u;
          }
        }
        if (!ok) break;
      }
      if (issued) {  // every MMA of this launch has completed before TMEM can be freed
        mma_commit_pair(drain_bar);
        mbar_drain(drain_bar, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else if (kFused && warp == 7) {
    if (lane == 0 && leader) {
      // ---------------- T generation (even CTA): D = Q^T U per stage of a fused item, into one of
      // TGEN_BUFS TMEM buffers.  Its commits track only these MMAs, so a T tile is ready as soon
      // as its own products are, however many statistics MMAs are queued.
      uint32_t tg = 0, qc = 0, gi = 0;
      uint32_t cu[STAGES] = {0, 0, 0, 0};  // fused uses of each stage (u_full phases)
      bool ok = true, issued = false;
      const uint32_t qsb = uint32_t(fz.rp) * 16u;
      const uint32_t u_lo = uint32_t(U_ROWS) * uint32_t(fz.rp) * 2u;
      const uint32_t q_base = smem_u32(qbuf);
      for (int it = cid; it < total_items && ok; it += ncl) {
        const Item w = decode(g, it);
        if (!fused_cross(w)) {
          gi += uint32_t(nkb);
          continue;
        }
        // the item's TMEM is free (the MMA thread has seen the last accumulators read) and its
        // Q^T is in shared memory
        if (!mbar_wait_cluster(tg_go, qc & 1u, wc) || !mbar_wait_cluster(q_full, qc & 1u, wc)) {
          ok = false;
          break;
        }
        fence_after();
        for (int kb = 0; kb < nkb && ok; ++kb) {
          const int s = int((gi + uint32_t(kb)) % STAGES);
          const uint32_t b = tg % TGEN_BUFS;
          const uint32_t par = ((tg / TGEN_BUFS) & 1u) ^ 1u;
          if ((!mbar_try_wait_cluster(u_full(s), cu[s] & 1u) && !mbar_wait_cluster(u_full(s), cu[s] & 1u, wc)) ||
              (!mbar_try_wait_cluster(tgen_empty(b), par) && !mbar_wait_cluster(tgen_empty(b), par, wc))) {
            ok = false;
            break;
          }
          ++cu[s];
          fence_after();
          const uint32_t u_base = smem_base + uint32_t(s) * STAGE_BYTES + A_BYTES;
          const uint32_t dt = tmem_base + TGEN_COL + b * uint32_t(BK);
          for (int ks = 0; ks < fz.rp / 16; ++ks) {
            const uint32_t ko = uint32_t(ks) * 256u;  // 16 k = two core matrices
            const uint64_t qh = sdesc(q_base + ko, 128u, qsb, kSwizzleNone);
            const uint64_t ql = sdesc(q_base + 8192u + ko, 128u, qsb, kSwizzleNone);
            const uint64_t uh = sdesc(u_base + ko, 128u, qsb, kSwizzleNone);
            const uint64_t ul = sdesc(u_base + u_lo + ko, 128u, qsb, kSwizzleNone);
            mma_f16_pair(dt, qh, uh, IDESC_TGEN, ks > 0 ? 1u : 0u);
            mma_f16_pair(dt, qh, ul, IDESC_TGEN, 1u);
            mma_f16_pair(dt, ql, uh, IDESC_TGEN, 1u);
          }
          issued = true;
          mma_commit_pair_mc(tgen_full(b), 0x3);
          mma_commit_pair_mc(u_free(s), 0x3);  // the stage's U has been read
          ++tg;
        }
        if (!ok) break;
        mma_commit_pair_mc(q_free, 0x3);  // every T generation of this item has read Q^T
        ++qc;
        gi += uint32_t(nkb);
      }
      if (issued) {  // these MMAs have completed before TMEM can be freed
        mma_commit_pair(tg_drain);
        mbar_drain(tg_drain, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else if (kFused && warp >= 8) {
    // ---------------- T conversion, second half of the tokens (warps 8..11, lane quarter warp % 4)
    const int q = warp & 3;
    uint32_t gi = 0, tg = 0, fc = 0;
    bool go = true;
    for (int it = cid; it < total_items && go; it += ncl) {
      const Item w = decode(g, it);
      if (fused_cross(w)) {
        // the MMA thread has seen every earlier item's statistics complete
        const bool okg = mbar_wait_cluster(tg_go, fc & 1u, wc);
        if (!__all_sync(0xffffffffu, okg)) break;
        ++fc;
        for (int kb = 0; kb < nkb; ++kb) {
          if (!convert_t(q, BK / 2, tg, gi + uint32_t(kb))) {
            go = false;
            break;
          }
          ++tg;
        }
      }
      gi += uint32_t(nkb);
    }
  } else if (kFused && warp == 6) {
    // ---------------- U and Q^T producer (both CTAs, fused cross items)
    int stage = 0;
    uint32_t qc = 0;
    uint32_t ucu[STAGES] = {0, 0, 0, 0};  // fused cross uses of each stage
    uint32_t ugo[STAGES] = {0, 0, 0, 0};  // of those, uses in the first STAGES iterations of an item
    bool ok = true;
    const int rp = fz.rp, r = fz.r;
    const uint32_t q_full_even = leader ? q_full : mapa_shared(q_full, 0);
    for (int it = cid; it < total_items && ok; it += ncl) {
      const Item w = decode(g, it);
      const bool gen = fused_cross(w);
      if (gen) {
        // the previous fused item's T generations have read Q^T (warp-uniform decision)
        const bool okq = qc == 0 || mbar_wait_cluster(q_free, (qc - 1) & 1u, wc);
        if (!__all_sync(0xffffffffu, okq)) {
          ok = false;
          break;
        }
        const float* Ql = fz.Q + int64_t(w.l) * r * g.d;
        __nv_bfloat16* qh = reinterpret_cast<__nv_bfloat16*>(qbuf);
        __nv_bfloat16* ql = reinterpret_cast<__nv_bfloat16*>(qbuf + 8192);
        for (int i = 0; i < BMC / 32; ++i) {
          const int cl = lane + 32 * i;  // channel of this CTA's 128
          const int c = w.mt[0] * BMP + int(rank) * BMC + cl;
          for (int sidx = 0; sidx < rp; ++sidx) {
            const float q = (sidx < r && c < g.d && LOCA_CHECK(int64_t(w.l) * r * g.d + int64_t(sidx) * g.d + c,
                                                               int64_t(g.L) * r * g.d))
                                ? __ldg(Ql + int64_t(sidx) * g.d + c)
                                : 0.f;
            __nv_bfloat16 h, lo;
            split_bf16(q, h, lo);
            const uint32_t off = kmaj16_off(cl, sidx, rp) >> 1;
            if (!LOCA_CHECK(off, 4096)) continue;
            qh[off] = h;
            ql[off] = lo;
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (leader) mbar_arrive(q_full);
          else mbar_arrive_remote(q_full_even);
        }
        ++qc;
      }
      if (!gen) {  // stages of other items are not this warp's
        stage = int((uint32_t(stage) + uint32_t(nkb)) % STAGES);
        continue;
      }
      // this CTA's 32 token rows of U for a stage: rp / 8 chunks of 16 bytes per part and row
      const uint4* Uh = reinterpret_cast<const uint4*>(fz.Uh + int64_t(w.l) * g.N * rp);
      const uint4* Ul = reinterpret_cast<const uint4*>(fz.Ul + int64_t(w.l) * g.N * rp);
      const int nq = rp / 8;
      auto load_u = [&](int kb, uint4* h, uint4* lo) {
        const int64_t n = int64_t(kb) * BK + int64_t(rank) * U_ROWS + lane;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          const bool in = qq < nq && n < g.N && LOCA_CHECK(n * nq + qq, g.N * nq);
          h[qq] = in ? __ldg(Uh + n * nq + qq) : make_uint4(0, 0, 0, 0);
          lo[qq] = in ? __ldg(Ul + n * nq + qq) : make_uint4(0, 0, 0, 0);
        }
      };
      uint4 ch[4], cl[4];
      load_u(0, ch, cl);
      for (int kb = 0; kb < nkb; ++kb) {
        uint4 nh[4], nl[4];
        if (kb + 1 < nkb) load_u(kb + 1, nh, nl);  // in flight while this stage waits
        // the stage's second A region is free for this iteration's U: in the item's first STAGES
        // iterations once the TMA producer has seen the stage's previous use done (it may have
        // held an A tile of another item), later once the T generation that read the previous U
        // of this item has completed (nothing else reads that region in a fused item)
        const bool first = kb < STAGES;
        const bool okg = first ? mbar_wait_cluster(u_go(stage), ugo[stage] & 1u, wc)
                               : mbar_wait_cluster(u_free(stage), (ucu[stage] - 1u) & 1u, wc);
        if (!__all_sync(0xffffffffu, okg)) {
          ok = false;
          break;
        }
        if (first) ++ugo[stage];
        ++ucu[stage];
        uint8_t* ub = smem + stage * STAGE_BYTES + A_BYTES;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          if (qq < nq) {
            const uint32_t off = kmaj16_off(lane, qq * 8, rp);
            *reinterpret_cast<uint4*>(ub + off) = ch[qq];
            *reinterpret_cast<uint4*>(ub + U_ROWS * rp * 2 + off) = cl[qq];
          }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          if (leader) mbar_arrive(u_full(stage));
          else mbar_arrive_remote(mapa_shared(u_full(stage), 0));
        }
        if (++stage == STAGES) stage = 0;
#pragma unroll
        for (int qq = 0; qq < 4; ++qq) {
          ch[qq] = nh[qq];
          cl[qq] = nl[qq];
        }
      }
    }
  } else if (warp >= 2 && warp < 6) {
    // ---------------- epilogue: warps 2..5, TMEM lane quarter = warp % 4
    const int q = warp & 3;
    uint8_t* box0 = epi + (warp - 2) * (K::kBufs * EPI_BOX_BYTES);
    const uint32_t box0_s = smem_u32(box0);
    const uint32_t acc_empty_leader = leader ? acc_empty : mapa_shared(acc_empty, 0);
    uint32_t acc_phase = 0;
    uint32_t nbox = 0;  // boxes this warp has handed to the TMA unit
    uint32_t gi = 0, tg = 0, fc = 0;  // fused: pipeline iteration, T tiles converted, fused items
    bool go = true;
    for (int it = cid; it < total_items && go; it += ncl) {
      const Item w = decode(g, it);
      const float al = alpha[w.l];
      const bool gen = fused_cross(w);
      if (gen) {  // the MMA thread has seen every earlier item's statistics complete
        const bool okg = mbar_wait_cluster(tg_go, fc & 1u, wc);
        if (!__all_sync(0xffffffffu, okg)) break;
        ++fc;
      }
      for (int seg = 0; seg < nseg && go; ++seg) {
        if (gen) {
          // this segment's T tiles, first half of the tokens (warps 8..11 take the second)
          const int kb_end = (seg + 1) * seg_kb < nkb ? (seg + 1) * seg_kb : nkb;
          for (int kb = seg * seg_kb; kb < kb_end; ++kb) {
            if (!convert_t(q, 0, tg, gi + uint32_t(kb))) {
              go = false;
              break;
            }
            ++tg;
          }
          if (!go) break;
        }
        const bool ok = mbar_wait_cluster(acc_full, acc_phase, wc);
        if (!__all_sync(0xffffffffu, ok)) {  // warp-uniform decision, warp reconverged
          go = false;
          break;
        }
        fence_after();
        // the previous segment's additions to these boxes are complete: fixed order of additions
        if (lane == 0) bulk_wait_group0();
        __syncwarp();
        const bool store = zero_first && seg == 0;
        for (int s = 0; s < w.nslots; ++s) {
          const bool is_gram = w.kind[s] == 0;
          const CUtensorMap* omap = is_gram ? &tmG : &tmC;
          const float sc = is_gram ? 1.f : al;
          const int i0 = w.mt[s] * BMP + int(rank) * BMC + q * 32;
#pragma unroll 1
          for (int c = 0; c < BN / 32; ++c) {
            float v[32];
            tmem_ld32(tmem_base + (uint32_t(q * 32) << 16) + uint32_t(s * BN + c * 32), v);
            if (s == w.nslots - 1 && c == BN / 32 - 1) {
              // all of this warp's accumulator reads are done: the MMA may start the next segment
              fence_before();
              __syncwarp();
              if (lane == 0) {
                if (leader) mbar_arrive(acc_empty);
                else mbar_arrive_remote(acc_empty_leader);
              }
            }
            const int j0 = w.nt * BN + c * 32;
            if (i0 >= g.d || j0 >= g.d) continue;  // warp-uniform; partial boxes are clipped by the TMA unit
            const uint32_t buf = nbox % uint32_t(K::kBufs);
            if (lane == 0) {  // this buffer's previous box has been read
              if (K::kBufs == 1) bulk_wait_group_read0();
              else bulk_wait_group_read1();
            }
            __syncwarp();
            // row `lane` of the box: 8 chunks of 16 bytes, chunk u at position u ^ (lane & 7)
            float4* row = reinterpret_cast<float4*>(box0 + buf * EPI_BOX_BYTES + lane * 128);
#pragma unroll
            for (int u = 0; u < 8; ++u)
              row[u ^ (lane & 7)] = make_float4(sc * v[4 * u], sc * v[4 * u + 1], sc * v[4 * u + 2],
                                                sc * v[4 * u + 3]);
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
              const uint32_t src = box0_s + buf * EPI_BOX_BYTES;
              if (LOCA_REQUIRE(i0 >= 0 && j0 >= 0 && j0 % 4 == 0)) {
                if (store) tma_store_3d(omap, src, j0, i0, w.l);
                else tma_reduce_add_3d(omap, src, j0, i0, w.l);
              }
              bulk_commit_group();
            }
            ++nbox;
          }
        }
        acc_phase ^= 1u;
      }
      gi += uint32_t(nkb);
    }
    if (lane == 0) bulk_wait_group0();  // every box written before the CTA can leave
    __syncwarp();
  }

  fence_before();
  cluster_sync();  // every role has stopped; the odd CTA's issue count is visible
  fence_after();
  if (warp == 0 && lane == 0 && leader) {
    // Copies still in flight when a role gave up.  Iteration t of the pipeline uses stage
    // t % STAGES; the even CTA arms it (the bytes of both CTAs) and issues its half, the odd CTA
    // issues its half after its own wait for the stage.  The two CTAs issued n_even and n_odd
    // iterations, |n_even - n_odd| <= STAGES, and every iteration before the last STAGES of
    // max(n_even, n_odd) has landed (a later use of its stage waited for it).  Of those last ones,
    // an iteration the odd CTA never issued gets its bytes settled, an iteration only the odd CTA
    // issued gets armed with its bytes, and every one is waited for.  After a normal run both
    // counts are equal, every phase has completed and these waits return at once.
    const uint32_t n_even = iters_done;
    const uint32_t n_odd = *reinterpret_cast<volatile uint32_t*>(odd_issued);
    const uint32_t hi = n_even > n_odd ? n_even : n_odd;
    const uint32_t lo = hi > uint32_t(STAGES) ? hi - uint32_t(STAGES) : 0u;
    for (uint32_t t = lo; t < hi; ++t) {
      const int s = int(t % STAGES);
      const Item w = decode(g, cid + int(t / uint32_t(nkb)) * ncl);
      const uint32_t odd_bytes = item_bytes(w);
      if (t >= n_odd && t < n_even) mbar_complete_tx(full_bar(s), odd_bytes);
      else if (t >= n_even && t < n_odd) mbar_arrive_expect_tx(full_bar(s), odd_bytes);
      mbar_drain(full_bar(s), (t / STAGES) & 1u, kDrainLimitNs);
    }
  }
  fence_before();
  cluster_sync();  // no CTA leaves while its peer may still use its barriers, smem or TMEM
  fence_after();
  if (warp == 1) tmem_dealloc_pair(tmem_base, TMEM_COLS);
}

// Lower triangle of every Gram_l from its upper triangle: element (i, j), i > j, becomes (j, i).
// One 64 x 64 tile (bi, bj), bi >= bj, per CTA (256 threads) through a padded shared tile; rows are
// read and written as 16-byte vectors when d % 4 == 0 (each thread moves 4 consecutive columns).
constexpr int MIR_T = 64;

__global__ void __launch_bounds__(256) k_gram_mirror(float* __restrict__ gram, int d, int nt) {
  __shared__ float tile[MIR_T][MIR_T + 1];
  const int l = blockIdx.y;
  // triangular index t = bi (bi + 1) / 2 + bj, 0 <= bj <= bi < nt
  const int t = blockIdx.x;
  int bi = int((sqrtf(8.f * float(t) + 1.f) - 1.f) * 0.5f);
  while ((bi + 1) * (bi + 2) / 2 <= t) ++bi;
  while (bi * (bi + 1) / 2 > t) --bi;
  const int bj = t - bi * (bi + 1) / 2;
  (void)nt;
  float* G = gram + int64_t(l) * d * d;
  const bool vec = (d & 3) == 0;
  const int tc4 = (threadIdx.x & 15) * 4, ty = threadIdx.x >> 4;  // 4 columns, 16 rows per pass
  for (int r = ty; r < MIR_T; r += 16) {  // source rows of the upper tile (bj, bi)
    const int i = bj * MIR_T + r, j = bi * MIR_T + tc4;
    if (i >= d) continue;
    if (vec && j + 3 < d && LOCA_CHECK_SPAN(int64_t(i) * d + j, 4, int64_t(d) * d)) {
      const float4 v = *reinterpret_cast<const float4*>(G + int64_t(i) * d + j);
      tile[r][tc4] = v.x;
      tile[r][tc4 + 1] = v.y;
      tile[r][tc4 + 2] = v.z;
      tile[r][tc4 + 3] = v.w;
    } else {
      for (int q = 0; q < 4; ++q)
        if (j + q < d && LOCA_CHECK(int64_t(i) * d + j + q, int64_t(d) * d)) tile[r][tc4 + q] = G[int64_t(i) * d + j + q];
    }
  }
  __syncthreads();
  for (int r = ty; r < MIR_T; r += 16) {  // destination rows of the lower tile (bi, bj)
    const int i = bi * MIR_T + r, j = bj * MIR_T + tc4;
    if (i >= d) continue;
    const float4 v = make_float4(tile[tc4][r], tile[tc4 + 1][r], tile[tc4 + 2][r], tile[tc4 + 3][r]);
    if (vec && bi > bj && j + 3 < d && LOCA_CHECK_SPAN(int64_t(i) * d + j, 4, int64_t(d) * d)) {
      *reinterpret_cast<float4*>(G + int64_t(i) * d + j) = v;  // off the diagonal: all i > j
    } else {
      const float vv[4] = {v.x, v.y, v.z, v.w};
      for (int q = 0; q < 4; ++q)
        if (j + q < d && i > j + q && LOCA_CHECK(int64_t(i) * d + j + q, int64_t(d) * d)) G[int64_t(i) * d + j + q] = vv[q];
    }
  }
}

// ------------------------------------------------------------------ host side
// 3-D view (channel, token, block) of X or T; boxes of 64 channels x BK tokens.
bool make_map(CUtensorMap* m, const void* base, int L, int64_t N, int64_t d) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(N), cuuint64_t(L)};
  cuuint64_t strides[2] = {cuuint64_t(d) * 2, cuuint64_t(N) * cuuint64_t(d) * 2};
  cuuint32_t box[3] = {64, BK, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 4-D view (64 channels, token, 64-channel block, block) of X or T, for d % 64 == 0: one box of
// `nblk` channel blocks x BK tokens lands as nblk consecutive 64 x BK swizzled tiles.
bool make_map_blocked(CUtensorMap* m, const void* base, int L, int64_t N, int64_t d, int nblk) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[4] = {64, cuuint64_t(N), cuuint64_t(d / 64), cuuint64_t(L)};
  cuuint64_t strides[3] = {cuuint64_t(d) * 2, 128, cuuint64_t(N) * cuuint64_t(d) * 2};
  cuuint32_t box[4] = {64, BK, cuuint32_t(nblk), 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D view (column, row, block) of the fp32 d x d outputs; boxes of 32 x 32 elements, 128-byte
// swizzle (the epilogue's staging layout).  Rows are d * 4 bytes (d % 8 == 0 on this path).
bool make_out_map(CUtensorMap* m, float* base, int L, int64_t d) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {cuuint64_t(d), cuuint64_t(d), cuuint64_t(L)};
  cuuint64_t strides[2] = {cuuint64_t(d) * 4, cuuint64_t(d) * cuuint64_t(d) * 4};
  cuuint32_t box[3] = {32, 32, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, static_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Clusters of 2 that can be resident at once (every SM pairs on GB300: 76 clusters on 152 SMs).
template <bool kFused>
int resident_clusters() {
  int clusters = sm_count() / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(2 * clusters));
  cfg.blockDim = dim3(Cfg<kFused>::kThreads);
  cfg.dynamicSmemBytes = Cfg<kFused>::kSmem;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k_gram_cross_tc<kFused>, &cfg) == cudaSuccess && n > 0 && n < clusters)
    clusters = n;
  cudaGetLastError();  // an unsupported query leaves the default
  return clusters;
}

// One launch of the statistics kernel (T from memory, or generated when fz.E != nullptr), then the
// mirror of the Gram's lower triangle.
template <bool kFused>
cudaError_t launch_stats(const void* X, const void* T, int L, int64_t N, int64_t d, const float* alpha,
                         int zero_first, float* gram, float* cross, int32_t* status, int32_t* abort_flag,
                         const Fuse& fz, cudaStream_t s) {
  CUtensorMap mx, mt, mxa, mta, mxb, mg, mc;
  memset(&mt, 0, sizeof(mt));
  memset(&mxa, 0, sizeof(mxa));
  memset(&mta, 0, sizeof(mta));
  memset(&mxb, 0, sizeof(mxb));
  if (!make_map(&mx, X, L, N, d) || (!kFused && !make_map(&mt, T, L, N, d)) || !make_out_map(&mg, gram, L, d) ||
      !make_out_map(&mc, cross, L, d))
    return cudaErrorInvalidValue;
  int blocked = 0;
  if (d % 64 == 0 && make_map_blocked(&mxa, X, L, N, d, BMC / 64) &&
      (kFused || make_map_blocked(&mta, T, L, N, d, BMC / 64)) && make_map_blocked(&mxb, X, L, N, d, BNC / 64))
    blocked = 1;
  Geo g;
  g.L = L;
  g.d = int(d);
  g.N = int(N);
  g.nM = int((d + BMP - 1) / BMP);
  g.nN = int((d + BN - 1) / BN);
  g.per_block = 0;
  g.full = 0;
  g.fused = kFused ? 1 : 0;
  for (int nt = 0; nt < g.nN; ++nt) g.per_block += items_of_col(g, nt);
  const int total = g.per_block * L;
  cudaError_t e = cudaFuncSetAttribute(k_gram_cross_tc<kFused>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg<kFused>::kSmem);
  if (e != cudaSuccess) return e;
  static int clusters_cached = 0;  // per process and variant; the library drives one device type
  if (clusters_cached == 0) clusters_cached = resident_clusters<kFused>();
  int clusters = clusters_cached;
  if (clusters > total) clusters = total;
  if (clusters < 1) clusters = 1;
  g.full = (g.per_block / clusters) * clusters;
  // abort flag and round counter (two int32 of the launch-local flag area)
  e = cudaMemsetAsync(abort_flag, 0, 2 * sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  // a round takes about nkb x 1024 tensor-core cycles; wait for the slowest cluster up to ~3x that
  const int64_t nkb = (N + BK - 1) / BK;
  const unsigned long long sync_ns = 50000ull + 2000ull * (unsigned long long)nkb;
  k_gram_cross_tc<kFused><<<2 * clusters, Cfg<kFused>::kThreads, Cfg<kFused>::kSmem, s>>>(
      mx, mt, mxa, mta, mxb, mg, mc, blocked, g, total, kSegTokens / BK, alpha, zero_first, status, abort_flag,
      reinterpret_cast<uint32_t*>(abort_flag + 1), wait_limit_ns(), sync_ns, fz);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int nt = int((d + MIR_T - 1) / MIR_T);
  k_gram_mirror<<<dim3(unsigned(nt * (nt + 1) / 2), unsigned(L)), 256, 0, s>>>(gram, int(d), nt);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gram_cross_tc(const void* X, const void* T, int L, int64_t N, int64_t d,
                                 const float* alpha, int zero_first, float* gram, float* cross,
                                 int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  const Fuse none{nullptr, nullptr, nullptr, 0, 0};
  return launch_stats<false>(X, T, L, N, d, alpha, zero_first, gram, cross, status, abort_flag, none, s);
}

int gram_fused_max_r() { return 32; }

size_t gram_fused_workspace_bytes(int L, int64_t N, int r) {
  const int rp = r <= 16 ? 16 : 32;
  return 256 + 2 * align256(sizeof(__nv_bfloat16) * size_t(L) * size_t(N) * size_t(rp));
}

cudaError_t launch_gram_cross_fused_tc(const void* X, const float* E, int C, const float* P, const float* Q,
                                       int r, int L, int64_t N, int64_t d, const float* alpha, int zero_first,
                                       float* gram, float* cross, int32_t* status, void* workspace,
                                       cudaStream_t s) {
  const int rp = r <= 16 ? 16 : 32;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  const size_t ub = align256(sizeof(__nv_bfloat16) * size_t(L) * size_t(N) * size_t(rp));
  __nv_bfloat16* Uh = reinterpret_cast<__nv_bfloat16*>(ws + 256);
  __nv_bfloat16* Ul = reinterpret_cast<__nv_bfloat16*>(ws + 256 + ub);
  k_fused_u<<<dim3(unsigned((N + 255) / 256), unsigned(L)), 256, 0, s>>>(E, N, C, P, r, rp, Uh, Ul);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const Fuse fz{Uh, Ul, Q, r, rp};
  return launch_stats<true>(X, nullptr, L, N, d, alpha, zero_first, gram, cross, status,
                            reinterpret_cast<int32_t*>(ws), fz, s);
}

}  // namespace loca
