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
constexpr int NUM_THREADS = 192;
constexpr int kSegTokens = 16384;                   // tokens per accumulation segment
constexpr int EPI_BOX_BYTES = 32 * 32 * 4;          // one 32-row x 32-column fp32 output box
constexpr int EPI_BUFS = 2;                         // staging boxes per epilogue warp
constexpr int EPI_BYTES = 4 * EPI_BUFS * EPI_BOX_BYTES;  // 32 KB
// barriers: full[S], empty[S], acc_full, acc_empty, drain
constexpr int NUM_BARS = 2 * STAGES + 3;
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + EPI_BYTES + 1024 /* align slack */ + 256 /* barriers */;
static_assert(SMEM_BYTES <= 232448, "shared memory per CTA");
static_assert(kSegTokens % (BK * kSyncEvery) == 0, "segments end on lockstep sync points");

// Instruction descriptor (kind::f16): D fp32, A bf16, B bf16, A and B MN-major, M = 256, N = 256.
constexpr uint32_t IDESC_PAIR = tc::idesc(1, 1, 1, 1, BMP, BN);

// ------------------------------------------------------------------ work items
struct Geo {
  int L, d, N;
  int nM, nN;       // 256-row tiles and 256-column tiles
  int per_block;    // work items per block l
  int full;         // items of each block that fill whole rounds of their own (0: plain order)
};

// Gram row tiles of column tile nt that contain an element with row <= column.
__device__ __host__ __forceinline__ int gram_rows(const Geo& g, int nt) {
  int last = nt * BN + BN - 1;
  if (last > g.d - 1) last = g.d - 1;
  int c = last / BMP + 1;
  return c < g.nM ? c : g.nM;
}
__device__ __host__ __forceinline__ int items_of_col(const Geo& g, int nt) {
  return (gram_rows(g, nt) + g.nM + 1) / 2;
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
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(NUM_THREADS, 1)
    k_gram_cross_tc(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmT,
                    const __grid_constant__ CUtensorMap tmXa, const __grid_constant__ CUtensorMap tmTa,
                    const __grid_constant__ CUtensorMap tmXb, const __grid_constant__ CUtensorMap tmG,
                    const __grid_constant__ CUtensorMap tmC, int blocked, Geo g, int total_items, int seg_kb,
                    const float* __restrict__ alpha, int zero_first, int32_t* status, int32_t* abort_flag,
                    uint32_t* round_ctr, unsigned long long limit_ns, unsigned long long sync_ns) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint8_t* epi = smem + STAGES * STAGE_BYTES;  // 1024-aligned: the boxes use the 128-byte swizzle
  uint64_t* bars = reinterpret_cast<uint64_t*>(epi + EPI_BYTES);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + NUM_BARS);
  uint32_t* odd_issued = tmem_slot + 1;  // even CTA: pipeline iterations the odd CTA issued
  const uint32_t smem_base = smem_u32(smem);
  const uint32_t bar_base = smem_u32(bars);
  auto full_bar = [&](int s) { return bar_base + 8u * s; };
  auto empty_bar = [&](int s) { return bar_base + 8u * (STAGES + s); };
  const uint32_t acc_full = bar_base + 8u * (2 * STAGES);
  const uint32_t acc_empty = bar_base + 8u * (2 * STAGES + 1);
  const uint32_t drain_bar = bar_base + 8u * (2 * STAGES + 2);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int cid = int(cluster_id_x());
  const int ncl = int(ncluster_x());
  const WaitCtl wc{status, abort_flag, limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(full_bar(s), 1);
      mbar_init(empty_bar(s), 1);
    }
    mbar_init(acc_full, 1);
    mbar_init(acc_empty, 8);  // lane 0 of the 4 epilogue warps of each CTA
    mbar_init(drain_bar, 1);
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
        const uint32_t bytes_one = uint32_t(w.nslots) * A_BYTES + B_BYTES;
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
          const uint32_t fb = mapa_shared(full_bar(stage), 0);
          const uint32_t st = smem_base + uint32_t(stage) * STAGE_BYTES;
          const uint32_t bdst = st + 2u * A_BYTES;
          const int tok = kb * BK;
          const int col0 = w.nt * BN + int(rank) * BNC;
          if (blocked) {
            for (int s = 0; s < w.nslots; ++s)
              tma_load_4d_pair(st + uint32_t(s) * A_BYTES, w.kind[s] == 0 ? &tmXa : &tmTa, fb, 0, tok,
                               (w.mt[s] * BMP + int(rank) * BMC) / 64, w.l);
            tma_load_4d_pair(bdst, &tmXb, fb, 0, tok, col0 / 64, w.l);
          } else {
            for (int s = 0; s < w.nslots; ++s) {
              const CUtensorMap* map = w.kind[s] == 0 ? &tmX : &tmT;
              const uint32_t dst = st + uint32_t(s) * A_BYTES;
              const int row0 = w.mt[s] * BMP + int(rank) * BMC;
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
      for (int it = cid; it < total_items && ok; it += ncl) {
        const Item w = decode(g, it);
        const bool two = w.nslots == 2;
        for (int kb = 0; kb < nkb; ++kb) {
          const int in_seg = kb % seg_kb;
          if (in_seg == 0) {  // a new segment: wait until the epilogue has read the accumulators
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
      }
      if (issued) {  // every MMA of this launch has completed before TMEM can be freed
        mma_commit_pair(drain_bar);
        mbar_drain(drain_bar, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else {
    // ---------------- epilogue: warps 2..5, TMEM lane quarter = warp % 4
    const int q = warp & 3;
    uint8_t* box0 = epi + (warp - 2) * (EPI_BUFS * EPI_BOX_BYTES);
    const uint32_t box0_s = smem_u32(box0);
    const uint32_t acc_empty_leader = leader ? acc_empty : mapa_shared(acc_empty, 0);
    uint32_t acc_phase = 0;
    uint32_t nbox = 0;  // boxes this warp has handed to the TMA unit
    bool go = true;
    for (int it = cid; it < total_items && go; it += ncl) {
      const Item w = decode(g, it);
      const float al = alpha[w.l];
      for (int seg = 0; seg < nseg; ++seg) {
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
            const uint32_t buf = nbox & (EPI_BUFS - 1);
            if (lane == 0) bulk_wait_group_read1();  // this buffer's previous box has been read
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
              if (store) tma_store_3d(omap, src, j0, i0, w.l);
              else tma_reduce_add_3d(omap, src, j0, i0, w.l);
              bulk_commit_group();
            }
            ++nbox;
          }
        }
        acc_phase ^= 1u;
      }
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
      const uint32_t odd_bytes = uint32_t(w.nslots) * A_BYTES + B_BYTES;
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
// One 32 x 32 tile (bi, bj), bi >= bj, per CTA (256 threads), through a padded shared tile.
__global__ void __launch_bounds__(256) k_gram_mirror(float* __restrict__ gram, int d, int nt) {
  __shared__ float tile[32][33];
  const int l = blockIdx.y;
  // triangular index t = bi (bi + 1) / 2 + bj, 0 <= bj <= bi < nt
  const int t = blockIdx.x;
  int bi = int((sqrtf(8.f * float(t) + 1.f) - 1.f) * 0.5f);
  while ((bi + 1) * (bi + 2) / 2 <= t) ++bi;
  while (bi * (bi + 1) / 2 > t) --bi;
  const int bj = t - bi * (bi + 1) / 2;
  (void)nt;
  float* G = gram + int64_t(l) * d * d;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  for (int r = ty; r < 32; r += 8) {  // source rows j of the upper tile (bj, bi)
    const int i = bj * 32 + r, j = bi * 32 + tx;
    if (i < d && j < d) tile[r][tx] = G[int64_t(i) * d + j];
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int i = bi * 32 + r, j = bj * 32 + tx;
    if (i < d && j < d && i > j) G[int64_t(i) * d + j] = tile[tx][r];
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
int resident_clusters() {
  int clusters = sm_count() / 2;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(unsigned(2 * clusters));
  cfg.blockDim = dim3(NUM_THREADS);
  cfg.dynamicSmemBytes = SMEM_BYTES;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeClusterDimension;
  at[0].val.clusterDim.x = 2;
  at[0].val.clusterDim.y = 1;
  at[0].val.clusterDim.z = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, k_gram_cross_tc, &cfg) == cudaSuccess && n > 0 && n < clusters)
    clusters = n;
  cudaGetLastError();  // an unsupported query leaves the default
  return clusters;
}

}  // namespace

cudaError_t launch_gram_cross_tc(const void* X, const void* T, int L, int64_t N, int64_t d,
                                 const float* alpha, int zero_first, float* gram, float* cross,
                                 int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  CUtensorMap mx, mt, mxa, mta, mxb, mg, mc;
  memset(&mxa, 0, sizeof(mxa));
  memset(&mta, 0, sizeof(mta));
  memset(&mxb, 0, sizeof(mxb));
  if (!make_map(&mx, X, L, N, d) || !make_map(&mt, T, L, N, d) || !make_out_map(&mg, gram, L, d) ||
      !make_out_map(&mc, cross, L, d))
    return cudaErrorInvalidValue;
  int blocked = 0;
  if (d % 64 == 0 && make_map_blocked(&mxa, X, L, N, d, BMC / 64) &&
      make_map_blocked(&mta, T, L, N, d, BMC / 64) && make_map_blocked(&mxb, X, L, N, d, BNC / 64))
    blocked = 1;
  Geo g;
  g.L = L;
  g.d = int(d);
  g.N = int(N);
  g.nM = int((d + BMP - 1) / BMP);
  g.nN = int((d + BN - 1) / BN);
  g.per_block = 0;
  g.full = 0;
  for (int nt = 0; nt < g.nN; ++nt) g.per_block += items_of_col(g, nt);
  const int total = g.per_block * L;
  cudaError_t e = cudaFuncSetAttribute(k_gram_cross_tc, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       SMEM_BYTES);
  if (e != cudaSuccess) return e;
  static int clusters_cached = 0;  // per process; the library drives one device type
  if (clusters_cached == 0) clusters_cached = resident_clusters();
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
  k_gram_cross_tc<<<2 * clusters, NUM_THREADS, SMEM_BYTES, s>>>(
      mx, mt, mxa, mta, mxb, mg, mc, blocked, g, total, kSegTokens / BK, alpha, zero_first, status, abort_flag,
      reinterpret_cast<uint32_t*>(abort_flag + 1), wait_limit_ns(), sync_ns);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const int nt = int((d + 31) / 32);
  k_gram_mirror<<<dim3(unsigned(nt * (nt + 1) / 2), unsigned(L)), 256, 0, s>>>(gram, int(d), nt);
  return cudaGetLastError();
}

}  // namespace loca
