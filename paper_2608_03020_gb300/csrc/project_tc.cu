// Projected statistics on the tensor cores (Eq. 9, Theorem S6):  GA_l = Gram_l A_l and
// CA_l = Cross_l A_l (d x k each), the d x d by d x k contractions that the ridge solve reduces to
// k x k systems.
//
// The kernel reads Gram_l and Cross_l once (8 d^2 bytes per block) and is bound by that HBM read.
// In fp32 on the FMA pipes the product costs 2 d^2 k FMAs per block, more than the read at k = 32,
// so it runs on the tensor cores (kind::f16, fp16 operands) with a two-part split of each fp32
// value: in each 32-channel slab a tile row is scaled by a power of two s so that its largest
// magnitude lies in [2^14, 2^15), and y = s x is carried as hi = fp16(y) and lo = fp16(y - hi)
// (both rounded to nearest; y - hi is exact in fp32), so |y - hi - lo| <= 2^-22 |y|, or 2^-25 for
// entries in fp16's subnormal range (2^-39 of the row's largest).  A_l's slab is split the same
// way with one power of two per column.  fp16 x fp16 products are exact in fp32, the tensor cores
// add in fp32, and the epilogue undoes both scales (exact multiplications by powers of two).
// Two MMAs per K-step, the tile's hi and lo parts against A's parts stacked as B (N = 2 KN), give
// all four part products.  The tensor cores drop a fraction of an ulp of the running sum at every
// step, always the same way, so the accumulator restarts at every 32-channel slab (4 MMAs) and the
// epilogue adds the slabs' products in fp32 with rounding to nearest, one row per thread: the
// result is as accurate as an fp32 FMA evaluation.  A tcgen05 MMA with N <= 128 costs about as
// much as one with N = 128, and every byte of a slab passes through shared memory several times
// (TMA write, split read and write, MMA operand reads), so two parts instead of three cut both.
//
// k_project_prep splits A_l once per launch: per (block, slab) a record with the scaled hi / lo
// parts of the 32 x k slab in the B operand's layout and the k reciprocal column scales.
//
// Work item = 128 rows of the stacked [Gram_l; Cross_l] (2 d rows per block) over all d columns.
// Persistent, one CTA per SM, 512 threads, four rings so that no role waits on another's latency:
//   warp 0      TMA producer: per K-slab a 128 x 32 fp32 tile of the matrix (128-byte swizzle) and
//               A's record for the slab (bulk copy) into a raw stage (PT_RAW stages).
//   split warps 8, 2, 3, 14 and 12, 10, 11, 15: two groups of four taking turns over the stages:
//               split a raw stage's tile into a split buffer (PT_SPLIT buffers, two per group), one
//               row per thread (K-major, no swizzle: 8-row x 16-byte core matrices), copy A's parts
//               beside it, and write the row and column scales into the scale slot of the stage's
//               accumulator.  The raw stage is released as soon as its values are in registers.
//               PT_RAW, PT_SPLIT and PT_ACC are multiples of the group count, so every use of a
//               stage, buffer or slot falls to the same group (each barrier phase a group waits
//               for follows one it has seen; a parity wait tells only consecutive phases apart).
//               No split warp shares the MMA warp's scheduler (warp % 4 == 1): issuing the MMAs
//               takes about half of that scheduler's cycles (warps 9 and 13 stay idle).
//   warp 1      owns the TMEM accumulators (PT_ACC of 128 lanes x 2 KN columns) and issues the
//               MMAs (kind::f16, M = 128, N = 2 KN, K = 16), one accumulator per K-slab.
//   warps 4-7   read each slab's accumulator (TMEM lane quarter warp % 4) and its scales, add the
//               two column groups, undo the scales into their rows' fp32 sums, and write the rows at
//               the end of the item.
// All waits are bounded (tc_ptx.cuh); a wait that gives up sets the status word, the other roles
// follow through the launch's abort flag, copies and MMAs in flight land before TMEM is freed.
// The bounded wait is an out-of-line call (registers saved around it), so each wait tries the
// barrier inline first.
#include <cuda_fp16.h>

#include <cstring>

#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

using namespace tc;

constexpr int PT_THREADS = 512;
constexpr int PT_RAW = 6;     // raw stages (TMA in flight)
constexpr int PT_SPLIT = 4;   // split buffers (MMA operands)
constexpr int PT_ACC = 4;     // TMEM accumulators and scale slots
constexpr int PT_CONV_WARPS = 8;
constexpr int PT_GROUPS = 2;  // split groups: group g takes the stages t with t % PT_GROUPS == g
constexpr int PT_GROUP_WARPS = PT_CONV_WARPS / PT_GROUPS;
static_assert(PT_CONV_WARPS % PT_GROUPS == 0, "whole groups");
static_assert(PT_RAW % PT_GROUPS == 0 && PT_SPLIT % PT_GROUPS == 0 && PT_ACC % PT_GROUPS == 0,
              "every use of a raw stage, split buffer or scale slot falls to one group");
constexpr int PT_TM = 128;    // rows per work item (TMEM lanes)
constexpr int PT_BK = 32;     // channels per K-slab (128 bytes of fp32: one swizzle row)
constexpr uint32_t PT_TILE = PT_TM * PT_BK * 4;   // 16 KB fp32 tile
constexpr uint32_t PT_PART = PT_TM * PT_BK * 2;   // 8 KB: one fp16 part of the tile

// K-major, no-swizzle 16-bit tile with 32 K columns: 8-row x 16-byte core matrices, K-adjacent
// ones 128 bytes apart, 8-row groups 512 bytes apart.  Byte offset of (row r, 8-column group u).
__host__ __device__ __forceinline__ uint32_t kmaj_chunk(int r, int u) {
  return uint32_t(r >> 3) * 512u + uint32_t(u) * 128u + uint32_t(r & 7) * 16u;
}

// A's record per (block, slab): rows 0 .. KN-1 the hi parts of the KN scaled columns, rows
// KN .. 2 KN-1 the lo parts (kmaj_chunk layout, 64 bytes per row), then KN reciprocal column
// scales (fp32; 0 for the padding columns s >= k).
template <int KN>
struct ARec {
  static constexpr uint32_t parts = 2u * KN * PT_BK * 2u;
  static constexpr uint32_t bytes = parts + KN * 4u;
  static_assert(bytes % 16 == 0, "bulk copies move multiples of 16 bytes");
};

// Byte offsets (the TMA tile 1024-byte aligned for the 128-byte swizzle).
template <int KN>
struct PtLayout {
  static constexpr int NB = 2 * KN;                          // B rows: A's parts hi, lo
  static constexpr uint32_t TMEM_COLS = PT_ACC * NB <= 256 ? 256u : 512u;
  static constexpr uint32_t arec_off = PT_TILE;              // in a raw stage: A's record
  static constexpr uint32_t raw_bytes = (PT_TILE + ARec<KN>::bytes + 1023u) & ~1023u;
  static constexpr uint32_t b_off = 2 * PT_PART;             // in a split buffer: hi, lo, A's parts
  static constexpr uint32_t split_bytes = b_off + ARec<KN>::parts;
  static constexpr uint32_t slot_floats = PT_TM + KN;         // row scales, then column scales
  static constexpr uint32_t split_base = PT_RAW * raw_bytes;
  static constexpr uint32_t slot_base = split_base + PT_SPLIT * split_bytes;
  static constexpr uint32_t bar_base = slot_base + PT_ACC * slot_floats * 4u;
  static constexpr uint32_t smem_bytes = bar_base + 512 + 1024;  // + barriers, alignment slack
  static_assert(raw_bytes % 1024 == 0 && split_bytes % 1024 == 0 && bar_base % 8 == 0,
                "tiles stay 1024-byte aligned, barriers 8-byte aligned");
  static_assert(PT_ACC * NB <= 512, "accumulators fit in TMEM");
  static_assert(smem_bytes <= 232448, "fits the 227 KB of shared memory a CTA may use");
};

struct PtGeo {
  int L, k;
  int64_t d;
  int nrt;    // 128-row tiles per matrix
  int nkb;    // K-slabs
  int items;  // L * 2 * nrt
};

__device__ __forceinline__ void pt_decode(const PtGeo& g, int it, int& l, int& which, int& row0) {
  l = it / (2 * g.nrt);
  const int rem = it - l * 2 * g.nrt;
  which = rem / g.nrt;                 // 0: Gram_l, 1: Cross_l
  row0 = (rem - which * g.nrt) * PT_TM;
}

// Power-of-two exponent e with m 2^e in [2^14, 2^15) for m = the largest magnitude of a row or
// column, clamped to [-126, 126] so that 2^e and 2^-e are normal fp32 numbers; 0 for m = 0 or a
// non-finite m; 126 for an fp32-subnormal m.
__device__ __forceinline__ int pt_shift(float m) {
  const int be = int((__float_as_uint(m) >> 23) & 0xffu);
  if (be == 255 || m == 0.f) return 0;
  if (be == 0) return 126;
  const int e = 141 - be;  // 14 - floor(log2 m)
  return e < -126 ? -126 : (e > 126 ? 126 : e);
}
__device__ __forceinline__ float pow2f(int e) { return __uint_as_float(uint32_t(e + 127) << 23); }

__device__ __forceinline__ uint32_t h2bits(__half2 h) { return *reinterpret_cast<const uint32_t*>(&h); }

// y[0..7] (already scaled) -> two 16-byte rows of fp16 parts, y ~ hi + lo (round to nearest at
// each step; y - hi is exact in fp32).
__device__ __forceinline__ void split8h(const float* y, uint4& hi, uint4& lo) {
  uint32_t h[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const __half2 hh = __floats2half2_rn(y[2 * i], y[2 * i + 1]);
    const float2 hf = __half22float2(hh);
    h[i] = h2bits(hh);
    l[i] = h2bits(__floats2half2_rn(y[2 * i] - hf.x, y[2 * i + 1] - hf.y));
  }
  hi = make_uint4(h[0], h[1], h[2], h[3]);
  lo = make_uint4(l[0], l[1], l[2], l[3]);
}

// A's records: thread (slab kb, column s) of block l splits A_l[32 kb .. 32 kb + 31, s].
constexpr int PP_THREADS = 128;
template <int KN>
__global__ void __launch_bounds__(PP_THREADS) k_project_prep(const float* __restrict__ A, int64_t d, int k,
                                                            int nkb, uint8_t* __restrict__ rec) {
  constexpr int SPB = PP_THREADS / KN;  // slabs per block
  const int l = blockIdx.y;
  const int kb = blockIdx.x * SPB + int(threadIdx.x) / KN;
  const int s = int(threadIdx.x) % KN;
  if (kb >= nkb) return;
  const float* Al = A + int64_t(l) * d * k;
  float a[PT_BK];
  float m = 0.f;
#pragma unroll
  for (int c = 0; c < PT_BK; ++c) {
    const int64_t ch = int64_t(kb) * PT_BK + c;
    a[c] = (s < k && ch < d) ? Al[ch * k + s] : 0.f;
    m = fmaxf(m, fabsf(a[c]));
  }
  const int e = pt_shift(m);
  const float sc = pow2f(e);
#pragma unroll
  for (int c = 0; c < PT_BK; ++c) a[c] *= sc;
  uint8_t* r = rec + (int64_t(l) * nkb + kb) * int64_t(ARec<KN>::bytes);
#pragma unroll
  for (int u = 0; u < PT_BK / 8; ++u) {
    uint4 hi, lo;
    split8h(a + 8 * u, hi, lo);
    *reinterpret_cast<uint4*>(r + kmaj_chunk(s, u)) = hi;
    *reinterpret_cast<uint4*>(r + kmaj_chunk(KN + s, u)) = lo;
  }
  reinterpret_cast<float*>(r + ARec<KN>::parts)[s] = s < k ? pow2f(-e) : 0.f;
}

template <int KN>
__global__ void __launch_bounds__(PT_THREADS, 1)
    k_project_tc(const __grid_constant__ CUtensorMap tmG, const __grid_constant__ CUtensorMap tmC,
                 const uint8_t* __restrict__ arec, PtGeo g, float* __restrict__ GA, float* __restrict__ CA,
                 int32_t* status, int32_t* abort_flag, unsigned long long limit_ns) {
  using PL = PtLayout<KN>;
  using AR = ARec<KN>;
  constexpr int NB = PL::NB;
  constexpr uint32_t ID = idesc(0, 0, 0, 0, PT_TM, NB);  // fp16 x fp16 -> fp32, both K-major
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const uint32_t sbase = smem_u32(smem);
  const uint32_t bar0 = sbase + PL::bar_base;
  auto raw_full = [&](int s) { return bar0 + 8u * s; };
  auto raw_empty = [&](int s) { return bar0 + 8u * (PT_RAW + s); };
  auto split_full = [&](int b) { return bar0 + 8u * (2 * PT_RAW + b); };
  auto split_empty = [&](int b) { return bar0 + 8u * (2 * PT_RAW + PT_SPLIT + b); };
  auto acc_full = [&](int a) { return bar0 + 8u * (2 * PT_RAW + 2 * PT_SPLIT + a); };
  auto acc_empty = [&](int a) { return bar0 + 8u * (2 * PT_RAW + 2 * PT_SPLIT + PT_ACC + a); };
  auto scale_full = [&](int a) { return bar0 + 8u * (2 * PT_RAW + 2 * PT_SPLIT + 2 * PT_ACC + a); };
  constexpr int NBAR = 2 * PT_RAW + 2 * PT_SPLIT + 3 * PT_ACC;
  const uint32_t drain_bar = bar0 + 8u * NBAR;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + PL::bar_base + 8u * (NBAR + 1));
  static_assert(8 * (NBAR + 2) <= 512, "barriers fit their 512 bytes");
  float* slots = reinterpret_cast<float*>(smem + PL::slot_base);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{status, abort_flag, limit_ns};

  if (threadIdx.x == 0) {
    for (int s = 0; s < PT_RAW; ++s) {
      mbar_init(raw_full(s), 1);
      mbar_init(raw_empty(s), PT_GROUP_WARPS);
    }
    for (int b = 0; b < PT_SPLIT; ++b) {
      mbar_init(split_full(b), PT_GROUP_WARPS);
      mbar_init(split_empty(b), 1);
    }
    for (int a = 0; a < PT_ACC; ++a) {
      mbar_init(acc_full(a), 1);
      mbar_init(acc_empty(a), 4);
      mbar_init(scale_full(a), PT_GROUP_WARPS);
    }
    mbar_init(drain_bar, 1);
    mbar_init_fence();
  }
  if (warp == 1) tmem_alloc(smem_u32(tmem_slot), PL::TMEM_COLS);
  fence_before();
  __syncthreads();
  fence_after();
  const uint32_t tmem_base = *tmem_slot;

  if (warp == 0) {
    // ---------------- TMA producer: the tile, then A's record for the slab
    if (lane == 0) {
      uint32_t t = 0, pending = 0, pending_par = 0;
      bool ok = true;
      for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
        int l, which, row0;
        pt_decode(g, it, l, which, row0);
        for (int kb = 0; kb < g.nkb; ++kb, ++t) {
          const int s = int(t % PT_RAW);
          const uint32_t ph = (t / PT_RAW) & 1u;
          if (!mbar_try_wait(raw_empty(s), ph ^ 1u) && !mbar_wait(raw_empty(s), ph ^ 1u, wc)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(raw_full(s), PT_TILE + AR::bytes);
          pending |= 1u << s;
          pending_par = (pending_par & ~(1u << s)) | (ph << s);
          const uint32_t st = sbase + uint32_t(s) * PL::raw_bytes;
          // x = kb * 32 fp32 = kb * 128 bytes: aligned for the tiled copy
          (void)LOCA_REQUIRE(kb * PT_BK * 4 % 16 == 0 && row0 >= 0);
          tma_load_3d(st, which ? &tmC : &tmG, raw_full(s), kb * PT_BK, row0, l);
          bulk_load(st + PL::arec_off, arec + (int64_t(l) * g.nkb + kb) * int64_t(AR::bytes), AR::bytes,
                    raw_full(s));
        }
      }
      if (!ok)
        for (int s = 0; s < PT_RAW; ++s)
          if (pending & (1u << s)) mbar_drain(raw_full(s), (pending_par >> s) & 1u, kDrainLimitNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer: per K-slab two K-steps of 16, the tile's two parts each
    if (lane == 0) {
      uint32_t t = 0;
      bool ok = true, issued = false;
      for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
        for (int kb = 0; kb < g.nkb; ++kb, ++t) {
          const int b = int(t % PT_SPLIT);
          const int a = int(t % PT_ACC);
          const uint32_t pa = ((t / PT_ACC) & 1u) ^ 1u, pb = (t / PT_SPLIT) & 1u;
          if ((!mbar_try_wait(acc_empty(a), pa) && !mbar_wait(acc_empty(a), pa, wc)) ||
              (!mbar_try_wait(split_full(b), pb) && !mbar_wait(split_full(b), pb, wc))) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t sp = sbase + PL::split_base + uint32_t(b) * PL::split_bytes;
          const uint32_t d_tmem = tmem_base + uint32_t(a * NB);
#pragma unroll
          for (int kk = 0; kk < PT_BK / 16; ++kk) {  // K = 16 fp16 = two core matrices along K
            const uint64_t bd = sdesc(sp + PL::b_off + uint32_t(kk) * 256u, 128u, 512u, kSwizzleNone);
#pragma unroll
            for (int p = 0; p < 2; ++p) {
              const uint64_t ad = sdesc(sp + uint32_t(p) * PT_PART + uint32_t(kk) * 256u, 128u, 512u, kSwizzleNone);
              mma_f16(d_tmem, ad, bd, ID, (kk | p) != 0 ? 1u : 0u);
            }
          }
          issued = true;
          mma_commit(split_empty(b));
          mma_commit(acc_full(a));
        }
      }
      if (!ok && issued) {
        mma_commit(drain_bar);
        mbar_drain(drain_bar, 0, kDrainLimitNs);
      }
    }
    __syncwarp();
  } else if (warp >= 4 && warp < 8) {
    // ---------------- warps 4..7: each slab's two column groups, unscaled, into the rows' sums
    const int q = warp & 3;  // TMEM lane quarter: rows q * 32 + lane of the item
    const uint32_t lane_base = uint32_t(q * 32) << 16;
    uint32_t t = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
      int l, which, row0;
      pt_decode(g, it, l, which, row0);
      float sum[KN];
#pragma unroll
      for (int i = 0; i < KN; ++i) sum[i] = 0.f;
      for (int kb = 0; kb < g.nkb; ++kb, ++t) {
        const int a = int(t % PT_ACC);
        const uint32_t pa = (t / PT_ACC) & 1u;
        const bool w_ok = (mbar_try_wait(acc_full(a), pa) || mbar_wait(acc_full(a), pa, wc)) &&
                          (mbar_try_wait(scale_full(a), pa) || mbar_wait(scale_full(a), pa, wc));
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        fence_after();
        const uint32_t ta = tmem_base + lane_base + uint32_t(a * NB);
        // columns [0, KN): products with A's hi part, [KN, 2 KN): with its lo part
        float v[NB];
        if constexpr (KN == 16) {
          tmem_ld32(ta, v);
        } else {
          tmem_ld32x2(ta, v);
        }
        // the two scales are undone one at a time (each product stays in fp32's range whenever the
        // result is); the slot's column scales are read here, before the slot is released
        const float* sl = slots + a * PL::slot_floats;
        const float inv_r = sl[q * 32 + lane];
#pragma unroll
        for (int i = 0; i < KN; ++i) sum[i] += ((v[i] + v[KN + i]) * inv_r) * sl[PT_TM + i];
        fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(acc_empty(a));  // the accumulator and the scale slot
      }
      if (!ok) break;
      const int64_t rr = int64_t(row0) + q * 32 + lane;
      if (rr < g.d && LOCA_CHECK_SPAN((int64_t(l) * g.d + rr) * g.k, g.k, int64_t(g.L) * g.d * g.k)) {
        float* out = (which ? CA : GA) + (int64_t(l) * g.d + rr) * g.k;  // k % 4 == 0: 16-byte rows
#pragma unroll
        for (int s4 = 0; s4 < KN; s4 += 4)
          if (s4 < g.k)
            *reinterpret_cast<float4*>(out + s4) = make_float4(sum[s4], sum[s4 + 1], sum[s4 + 2], sum[s4 + 3]);
      }
    }
  } else if (warp != 9 && warp != 13) {
    // ---------------- split warps (not on the MMA warp's scheduler): the groups take turns, so that
    // one stage's split latency overlaps the next one's; each group has a warp on schedulers 0, 2, 3
    const int cw = warp == 8 ? 0 : warp == 2 ? 1 : warp == 3 ? 2 : warp == 14 ? 3
                 : warp == 12 ? 4 : warp == 10 ? 5 : warp == 11 ? 6 : 7;  // warp 15
    const int grp = cw / PT_GROUP_WARPS;
    const int ct = (cw % PT_GROUP_WARPS) * 32 + lane;  // thread within the group: tile row ct
    constexpr int NT = PT_GROUP_WARPS * 32;
    static_assert(NT == PT_TM, "one tile row per thread of a group");
    constexpr int CPY = int(AR::parts / 16);        // 16-byte chunks of A's parts
    constexpr int CPT = (CPY + NT - 1) / NT;
    const int r = ct;
    uint32_t t = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
      for (int kb = 0; kb < g.nkb; ++kb, ++t) {
        if (int(t % PT_GROUPS) != grp) continue;
        const int s = int(t % PT_RAW);
        const int b = int(t % PT_SPLIT);
        const int a = int(t % PT_ACC);
        // raw stage, split buffer and scale slot: this group's only (see the static_assert), each
        // released in order; the slot is free once the epilogue released stage t - PT_ACC
        const uint32_t pr = (t / PT_RAW) & 1u, pb = ((t / PT_SPLIT) & 1u) ^ 1u, pa = ((t / PT_ACC) & 1u) ^ 1u;
        bool w_ok = mbar_try_wait(raw_full(s), pr) || mbar_wait(raw_full(s), pr, wc);
        w_ok = w_ok && (mbar_try_wait(split_empty(b), pb) || mbar_wait(split_empty(b), pb, wc));
        w_ok = w_ok && (mbar_try_wait(acc_empty(a), pa) || mbar_wait(acc_empty(a), pa, wc));
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        const uint8_t* rp = smem + uint32_t(s) * PL::raw_bytes;
        uint8_t* sp = smem + PL::split_base + uint32_t(b) * PL::split_bytes;
        // read everything this thread needs from the raw stage first: row r is the 8 raw 16-byte
        // chunks c at positions c ^ (r % 8) (128-byte swizzle); then A's parts and column scale
        float x[PT_BK];
        const uint8_t* row = rp + uint32_t(r) * 128u;
#pragma unroll
        for (int c = 0; c < PT_BK / 4; ++c) {
          const float4 v4 = *reinterpret_cast<const float4*>(row + ((uint32_t(c) ^ uint32_t(r & 7)) << 4));
          x[4 * c] = v4.x;
          x[4 * c + 1] = v4.y;
          x[4 * c + 2] = v4.z;
          x[4 * c + 3] = v4.w;
        }
        uint4 ap[CPT];
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          const int c = ct + j * NT;
          ap[j] = c < CPY ? *reinterpret_cast<const uint4*>(rp + PL::arec_off + 16u * uint32_t(c)) : make_uint4(0, 0, 0, 0);
        }
        const float inv_col = ct < KN ? reinterpret_cast<const float*>(rp + PL::arec_off + AR::parts)[ct] : 0.f;
        // every raw value is in registers: the stage may be refilled
        __syncwarp();
        if (lane == 0) mbar_arrive(raw_empty(s));
        float m = 0.f;
#pragma unroll
        for (int c = 0; c < PT_BK; ++c) m = fmaxf(m, fabsf(x[c]));
        const int e = pt_shift(m);
        const float sc = pow2f(e);
#pragma unroll
        for (int c = 0; c < PT_BK; ++c) x[c] *= sc;
#pragma unroll
        for (int u = 0; u < PT_BK / 8; ++u) {
          uint4 hi, lo;
          split8h(x + 8 * u, hi, lo);
          const uint32_t off = kmaj_chunk(r, u);
          if (!LOCA_CHECK_SPAN(off, 16, PT_PART)) continue;
          *reinterpret_cast<uint4*>(sp + off) = hi;
          *reinterpret_cast<uint4*>(sp + PT_PART + off) = lo;
        }
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
          const int c = ct + j * NT;
          if (c < CPY) *reinterpret_cast<uint4*>(sp + PL::b_off + 16u * uint32_t(c)) = ap[j];
        }
        float* sl = slots + a * PL::slot_floats;
        sl[r] = pow2f(-e);
        if (ct < KN) sl[PT_TM + ct] = inv_col;
        fence_proxy_async_smem();  // the split tiles visible to the tensor cores
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(split_full(b));
          mbar_arrive(scale_full(a));
        }
      }
    }
  }

  fence_before();
  __syncthreads();
  fence_after();
  if (warp == 1) tmem_dealloc(tmem_base, PL::TMEM_COLS);
}

bool make_map_f32(CUtensorMap* m, const void* base, uint64_t inner, uint64_t rows, uint64_t outer, uint32_t box_x,
                  uint32_t box_y, bool swizzle) {
  auto fn = tensor_map_encoder();
  if (!fn) return false;
  cuuint64_t dims[3] = {cuuint64_t(inner), cuuint64_t(rows), cuuint64_t(outer)};
  cuuint64_t strides[2] = {cuuint64_t(inner) * 4, cuuint64_t(rows) * cuuint64_t(inner) * 4};
  cuuint32_t box[3] = {box_x, box_y, 1};
  cuuint32_t estr[3] = {1, 1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<void*>(base), dims, strides, box, estr,
            CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_NONE,
            CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int n_slabs(int64_t d) { return int((d + PT_BK - 1) / PT_BK); }

template <int KN>
cudaError_t launch_kn(const float* gram, const float* cross, const float* A, int L, int64_t d, int k, float* GA,
                      float* CA, void* arec, int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  CUtensorMap tmG, tmC;
  memset(&tmG, 0, sizeof(tmG));
  memset(&tmC, 0, sizeof(tmC));
  if (!make_map_f32(&tmG, gram, uint64_t(d), uint64_t(d), uint64_t(L), PT_BK, PT_TM, true) ||
      !make_map_f32(&tmC, cross, uint64_t(d), uint64_t(d), uint64_t(L), PT_BK, PT_TM, true))
    return cudaErrorInvalidValue;
  PtGeo g;
  g.L = L;
  g.k = k;
  g.d = d;
  g.nrt = int((d + PT_TM - 1) / PT_TM);
  g.nkb = n_slabs(d);
  g.items = L * 2 * g.nrt;
  constexpr int SPB = PP_THREADS / KN;
  k_project_prep<KN><<<dim3(unsigned((g.nkb + SPB - 1) / SPB), unsigned(L)), PP_THREADS, 0, s>>>(
      A, d, k, g.nkb, static_cast<uint8_t*>(arec));
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = cudaMemsetAsync(abort_flag, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  int grid = sm_count();
  if (grid > g.items) grid = g.items;
  const uint32_t shm = PtLayout<KN>::smem_bytes;
  e = cudaFuncSetAttribute(k_project_tc<KN>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
  if (e != cudaSuccess) return e;
  k_project_tc<KN><<<unsigned(grid), PT_THREADS, shm, s>>>(tmG, tmC, static_cast<const uint8_t*>(arec), g, GA, CA,
                                                           status, abort_flag, wait_limit_ns());
  return cudaGetLastError();
}

}  // namespace

bool project_tc_supported(const float* gram, const float* cross, const float* A, int64_t d, int k) {
  auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  return d % 4 == 0 && k % 4 == 0 && k >= 4 && k <= 32 && d < (int64_t(1) << 31) && a16(gram) && a16(cross) &&
         a16(A) && tensor_map_encoder() != nullptr;
}

size_t project_tc_workspace_bytes(int L, int64_t d, int k) {
  const size_t rec = k <= 16 ? ARec<16>::bytes : ARec<32>::bytes;
  return size_t(L) * size_t(n_slabs(d)) * rec;
}

cudaError_t launch_project_tc(const float* gram, const float* cross, const float* A, int L, int64_t d, int k,
                              float* GA, float* CA, void* arec, int32_t* status, int32_t* abort_flag,
                              cudaStream_t s) {
  if ((reinterpret_cast<uintptr_t>(arec) & 15u) != 0) return cudaErrorInvalidValue;
  if (k <= 16) return launch_kn<16>(gram, cross, A, L, d, k, GA, CA, arec, status, abort_flag, s);
  return launch_kn<32>(gram, cross, A, L, d, k, GA, CA, arec, status, abort_flag, s);
}

}  // namespace loca
