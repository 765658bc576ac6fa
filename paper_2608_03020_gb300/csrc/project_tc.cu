// Projected statistics on the tensor cores (Eq. 9, Theorem S6):  GA_l = Gram_l A_l and
// CA_l = Cross_l A_l (d x k each), the d x d by d x k contractions that the ridge solve reduces to
// k x k systems.
//
// The kernel reads Gram_l and Cross_l once (8 d^2 bytes per block) and is bound by that HBM read.
// In fp32 on the FMA pipes the product costs 2 d^2 k FMAs per block, more than the read at k = 32,
// so it runs on the tensor cores (kind::f16, bf16 operands) with an exact three-way split: every
// fp32 value x is hi + mid + lo with hi = bf16(x), mid = bf16(x - hi), lo = x - hi - mid (eight
// significant bits, a bf16 value), so the sum is x itself.  The split matrix tile is the A operand
// (M = 128 rows) and the split A_l slab, its three parts stacked, the B operand (N = 3 KN columns):
// three MMAs per K-step give all nine part products, each exact in fp32, and the epilogue adds the
// three column groups.  The tensor cores add in fp32 and drop a fraction of an ulp of the running
// sum at every step, always the same way; so the accumulator restarts at every K-slab of 32
// channels (6 MMAs) and the epilogue adds the slabs' partial products in fp32 with rounding to
// nearest, one row per thread, which keeps the result as accurate as an fp32 FMA evaluation.
// A tcgen05 MMA with N <= 128 costs about as much as one with N = 128, so the part count, not the
// width, sets the MMA time: 6 MMAs per 16 KB slab, under the slab's HBM time.
//
// Work item = 128 rows of the stacked [Gram_l; Cross_l] (2 d rows per block) over all d columns.
// Persistent, one CTA per SM, 512 threads, three rings so that no role waits on another's latency:
//   warp 0      TMA producer: per K-slab a 128 x 32 fp32 tile of the matrix (128-byte swizzle) and
//               the 32 x k rows of A_l (plain) into a raw stage (PT_RAW stages).
//   split warps 8, 2, 3, 14 and 12, 10, 11, 15: two groups of four taking turns over the stages:
//               split a raw stage into a split buffer (PT_SPLIT buffers, two per group): the
//               tile's hi / mid / lo bf16 parts and A's slab parts, all K-major without swizzle
//               (8-row x 16-byte core matrices); the raw stage is released as soon as its values
//               are in registers.  PT_RAW is a multiple of the group count, so every use of a
//               raw stage falls to the same group (each barrier phase a group waits for follows
//               one it has seen).
//               A stage's MMAs free its split buffer, so the split of stage t waits for the MMAs
//               of stage t - PT_SPLIT.  No split warp shares the MMA warp's scheduler
//               (warp % 4 == 1): issuing the MMAs takes about half of that scheduler's cycles,
//               and a split warp there was the one that set the pace (warps 9 and 13 stay idle).
//   warp 1      owns the TMEM accumulators (PT_ACC of 128 lanes x 3 KN columns) and issues the
//               MMAs (kind::f16, M = 128, N = 3 KN, K = 16), one accumulator per K-slab.
//   warps 4-7   read each slab's accumulator (TMEM lane quarter warp % 4), add its three column
//               groups into their rows' fp32 sums, and write the rows at the end of the item.
// All waits are bounded (tc_ptx.cuh); a wait that gives up sets the status word, the other roles
// follow through the launch's abort flag, copies and MMAs in flight land before TMEM is freed.
#include <cuda_bf16.h>

#include <cstring>

#include "loca_internal.h"
#include "tc_ptx.cuh"

namespace loca {
namespace {

using namespace tc;

constexpr int PT_THREADS = 512;
constexpr int PT_RAW = 4;     // raw stages (TMA in flight)
constexpr int PT_SPLIT = 4;   // split buffers (MMA operands)
constexpr int PT_ACC = 4;     // TMEM accumulators
constexpr int PT_CONV_WARPS = 8;
constexpr int PT_GROUPS = 2;  // split groups: group g takes the stages t with t % PT_GROUPS == g
constexpr int PT_GROUP_WARPS = PT_CONV_WARPS / PT_GROUPS;
static_assert(PT_CONV_WARPS % PT_GROUPS == 0 && PT_SPLIT % PT_GROUPS == 0, "groups own whole split buffers");
// Every use of a raw stage then falls to the same group, which takes its stages in order: an
// mbarrier parity wait tells only consecutive phases apart, so with an odd count a group running
// ahead could take the phase of the other group's earlier use (its copy still landing) for its own.
static_assert(PT_RAW % PT_GROUPS == 0, "groups own whole raw stages");
constexpr int PT_TM = 128;    // rows per work item (TMEM lanes)
constexpr int PT_BK = 32;     // channels per K-slab (128 bytes of fp32: one swizzle row)
constexpr uint32_t PT_TILE = PT_TM * PT_BK * 4;   // 16 KB fp32 tile
constexpr uint32_t PT_PART = PT_TM * PT_BK * 2;   // 8 KB: one bf16 part of the tile

// K-major, no-swizzle bf16 tile with 32 K columns: 8-row x 16-byte core matrices, K-adjacent
// ones 128 bytes apart, 8-row groups 512 bytes apart.  Byte offset of (row r, 8-column group u).
__device__ __forceinline__ uint32_t kmaj_chunk(int r, int u) {
  return uint32_t(r >> 3) * 512u + uint32_t(u) * 128u + uint32_t(r & 7) * 16u;
}

// Byte offsets (the TMA tile 1024-byte aligned for the 128-byte swizzle).
template <int KN>
struct PtLayout {
  static constexpr int NB = 3 * KN;                          // B rows: A's parts hi, mid, lo
  static constexpr uint32_t TMEM_COLS = PT_ACC * NB <= 256 ? 256u : 512u;
  static constexpr uint32_t araw_off = PT_TILE;              // in a raw stage: A rows, 32 x k fp32
  static constexpr uint32_t raw_bytes = PT_TILE + PT_BK * KN * 4;
  static constexpr uint32_t b_off = 3 * PT_PART;             // in a split buffer: parts at p * 8 KB
  static constexpr uint32_t split_bytes = b_off + NB * PT_BK * 2;
  static constexpr uint32_t split_base = PT_RAW * raw_bytes;
  static constexpr uint32_t bar_base = split_base + PT_SPLIT * split_bytes;
  static constexpr uint32_t smem_bytes = bar_base + 512 + 1024;  // + barriers, alignment slack
  static_assert(raw_bytes % 1024 == 0 && split_bytes % 1024 == 0, "tiles stay 1024-byte aligned");
  static_assert(PT_ACC * NB <= 512, "accumulators fit in TMEM");
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

__device__ __forceinline__ uint32_t bf16x2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}
__device__ __forceinline__ float bf16_lo_f(uint32_t p) { return __uint_as_float(p << 16); }
__device__ __forceinline__ float bf16_hi_f(uint32_t p) { return __uint_as_float(p & 0xffff0000u); }

// x[0..7] -> three 16-byte rows of bf16 parts with x = hi + mid + lo exactly (round to nearest at
// each step; each remainder is exact in fp32 and the last has at most eight significant bits).
__device__ __forceinline__ void split8(const float* x, uint4& hi, uint4& mid, uint4& lo) {
  uint32_t h[4], m[4], l[4];
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    h[i] = bf16x2(x[2 * i], x[2 * i + 1]);
    const float r0 = x[2 * i] - bf16_lo_f(h[i]);
    const float r1 = x[2 * i + 1] - bf16_hi_f(h[i]);
    m[i] = bf16x2(r0, r1);
    l[i] = bf16x2(r0 - bf16_lo_f(m[i]), r1 - bf16_hi_f(m[i]));
  }
  hi = make_uint4(h[0], h[1], h[2], h[3]);
  mid = make_uint4(m[0], m[1], m[2], m[3]);
  lo = make_uint4(l[0], l[1], l[2], l[3]);
}

template <int KN>
__global__ void __launch_bounds__(PT_THREADS, 1)
    k_project_tc(const __grid_constant__ CUtensorMap tmG, const __grid_constant__ CUtensorMap tmC,
                 const __grid_constant__ CUtensorMap tmA, PtGeo g, float* __restrict__ GA, float* __restrict__ CA,
                 int32_t* status, int32_t* abort_flag, unsigned long long limit_ns) {
  using PL = PtLayout<KN>;
  constexpr int NB = PL::NB;
  constexpr uint32_t ID = idesc(1, 1, 0, 0, PT_TM, NB);  // bf16 x bf16 -> fp32, both K-major
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
  const uint32_t drain_bar = bar0 + 8u * (2 * PT_RAW + 2 * PT_SPLIT + 2 * PT_ACC);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + PL::bar_base + 8u * (2 * PT_RAW + 2 * PT_SPLIT + 2 * PT_ACC + 1));
  static_assert(8 * (2 * PT_RAW + 2 * PT_SPLIT + 2 * PT_ACC + 2) <= 512, "barriers fit their 512 bytes");

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const WaitCtl wc{status, abort_flag, limit_ns};
  const uint32_t a_bytes = uint32_t(PT_BK) * uint32_t(g.k) * 4u;

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
    // ---------------- TMA producer
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
          mbar_arrive_expect_tx(raw_full(s), PT_TILE + a_bytes);
          pending |= 1u << s;
          pending_par = (pending_par & ~(1u << s)) | (ph << s);
          const uint32_t st = sbase + uint32_t(s) * PL::raw_bytes;
          // x = kb * 32 fp32 = kb * 128 bytes: aligned for the tiled copy
          (void)LOCA_REQUIRE(kb * PT_BK * 4 % 16 == 0 && row0 >= 0);
          tma_load_3d(st, which ? &tmC : &tmG, raw_full(s), kb * PT_BK, row0, l);
          tma_load_3d(st + PL::araw_off, &tmA, raw_full(s), 0, kb * PT_BK, l);
        }
      }
      if (!ok)
        for (int s = 0; s < PT_RAW; ++s)
          if (pending & (1u << s)) mbar_drain(raw_full(s), (pending_par >> s) & 1u, kDrainLimitNs);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ---------------- MMA issuer: per K-slab two K-steps of 16, three tile parts each
    if (lane == 0) {
      uint32_t t = 0;
      bool ok = true, issued = false;
      for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
        for (int kb = 0; kb < g.nkb; ++kb, ++t) {
          const int b = int(t % PT_SPLIT);
          const int a = int(t % PT_ACC);
          const uint32_t pa = ((t / PT_ACC) & 1u) ^ 1u;
          if (!mbar_try_wait(acc_empty(a), pa) && !mbar_wait(acc_empty(a), pa, wc)) { ok = false; break; }
          if (!mbar_try_wait(split_full(b), (t / PT_SPLIT) & 1u) &&
              !mbar_wait(split_full(b), (t / PT_SPLIT) & 1u, wc)) {
            ok = false;
            break;
          }
          fence_after();
          const uint32_t sp = sbase + PL::split_base + uint32_t(b) * PL::split_bytes;
          const uint32_t d_tmem = tmem_base + uint32_t(a * NB);
#pragma unroll
          for (int kk = 0; kk < PT_BK / 16; ++kk) {  // K = 16 bf16 = two core matrices along K
            const uint64_t bd = sdesc(sp + PL::b_off + uint32_t(kk) * 256u, 128u, 512u, kSwizzleNone);
#pragma unroll
            for (int p = 0; p < 3; ++p) {
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
    // ---------------- warps 4..7: each slab's three column groups into the rows' sums, then the rows
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
        const bool w_ok = mbar_try_wait(acc_full(a), pa) || mbar_wait(acc_full(a), pa, wc);
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        fence_after();
        const uint32_t ta = tmem_base + lane_base + uint32_t(a * NB);
        // columns [0, KN): products with A's hi part, [KN, 2 KN): mid, [2 KN, 3 KN): lo; the two
        // small groups are added first
        if constexpr (KN == 16) {
          float v[48];
          tmem_ld32(ta, v);
          tmem_ld16(ta + 32, v + 32);
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(acc_empty(a));
#pragma unroll
          for (int i = 0; i < 16; ++i) sum[i] += v[i] + (v[16 + i] + v[32 + i]);
        } else {
          float sm[32], v[32];
          tmem_ld32(ta + 32, sm);
          tmem_ld32(ta + 64, v);
#pragma unroll
          for (int i = 0; i < 32; ++i) sm[i] += v[i];
          tmem_ld32(ta, v);
          fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(acc_empty(a));
#pragma unroll
          for (int i = 0; i < 32; ++i) sum[i] += v[i] + sm[i];
        }
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
    const int ct = (cw % PT_GROUP_WARPS) * 32 + lane;  // thread within the group
    constexpr int NT = PT_GROUP_WARPS * 32;
    constexpr int UPT = PT_TM * (PT_BK / 8) / NT;  // 8-channel chunks of one row per thread
    static_assert(NT % PT_TM == 0 && UPT >= 1, "whole rows of chunks per thread");
    const int r = ct % PT_TM;                       // the tile row of this thread
    const int u0 = (ct / PT_TM) * UPT;              // its first 8-channel chunk
    uint32_t t = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < g.items && ok; it += gridDim.x) {
      for (int kb = 0; kb < g.nkb; ++kb, ++t) {
        if (int(t % PT_GROUPS) != grp) continue;
        const int s = int(t % PT_RAW);
        const int b = int(t % PT_SPLIT);
        // raw stage s: this group's stages only (PT_RAW % PT_GROUPS == 0), taken in order.  The
        // bounded wait is a call (registers saved around it), so an inline try_wait goes first.
        const uint32_t pr = (t / PT_RAW) & 1u, pb = ((t / PT_SPLIT) & 1u) ^ 1u;
        bool w_ok = mbar_try_wait(raw_full(s), pr) || mbar_wait(raw_full(s), pr, wc);
        w_ok = w_ok && (mbar_try_wait(split_empty(b), pb) || mbar_wait(split_empty(b), pb, wc));
        if (!__all_sync(0xffffffffu, w_ok)) {
          ok = false;
          break;
        }
        const uint8_t* rp = smem + uint32_t(s) * PL::raw_bytes;
        uint8_t* sp = smem + PL::split_base + uint32_t(b) * PL::split_bytes;
        // read everything this thread needs from the raw stage first: row r, channels 8u .. 8u + 7
        // are the raw 16-byte chunks 2u and 2u + 1 of the row, at positions (2u) ^ (r % 8) and
        // (2u + 1) ^ (r % 8) (128-byte swizzle); then A's values for the B rows
        float xv[UPT][8];
        const uint8_t* row = rp + uint32_t(r) * 128u;
#pragma unroll
        for (int j = 0; j < UPT; ++j) {
          const int u = u0 + j;
          const float4 x0 = *reinterpret_cast<const float4*>(row + ((uint32_t(2 * u) ^ uint32_t(r & 7)) << 4));
          const float4 x1 = *reinterpret_cast<const float4*>(row + ((uint32_t(2 * u + 1) ^ uint32_t(r & 7)) << 4));
          xv[j][0] = x0.x; xv[j][1] = x0.y; xv[j][2] = x0.z; xv[j][3] = x0.w;
          xv[j][4] = x1.x; xv[j][5] = x1.y; xv[j][6] = x1.z; xv[j][7] = x1.w;
        }
        // B rows p KN + s (part p of column s of A), channels 8u .. 8u + 7; columns s >= k are 0
        const float* araw = reinterpret_cast<const float*>(rp + PL::araw_off);
        constexpr int BPT = (KN * (PT_BK / 8) + NT - 1) / NT;
        float av[BPT][8];
#pragma unroll
        for (int j = 0; j < BPT; ++j) {
          const int c = ct + j * NT;
          const int sc = c % KN, u = c / KN;
#pragma unroll
          for (int e = 0; e < 8; ++e)
            av[j][e] = (c < KN * (PT_BK / 8) && sc < g.k) ? araw[(8 * u + e) * g.k + sc] : 0.f;
        }
        uint4 h[UPT], m[UPT], lo[UPT];
#pragma unroll
        for (int j = 0; j < UPT; ++j) split8(xv[j], h[j], m[j], lo[j]);
        uint4 bh[BPT], bm[BPT], bl[BPT];
#pragma unroll
        for (int j = 0; j < BPT; ++j) split8(av[j], bh[j], bm[j], bl[j]);
        // every raw value is consumed: the stage may be refilled
        __syncwarp();
        if (lane == 0) mbar_arrive(raw_empty(s));
#pragma unroll
        for (int j = 0; j < UPT; ++j) {
          const uint32_t off = kmaj_chunk(r, u0 + j);
          if (!LOCA_CHECK_SPAN(off, 16, PT_PART)) continue;
          *reinterpret_cast<uint4*>(sp + off) = h[j];
          *reinterpret_cast<uint4*>(sp + PT_PART + off) = m[j];
          *reinterpret_cast<uint4*>(sp + 2 * PT_PART + off) = lo[j];
        }
#pragma unroll
        for (int j = 0; j < BPT; ++j) {
          const int c = ct + j * NT;
          if (c >= KN * (PT_BK / 8)) continue;
          const int sc = c % KN, u = c / KN;
          const uint32_t o0 = kmaj_chunk(sc, u), o1 = kmaj_chunk(KN + sc, u), o2 = kmaj_chunk(2 * KN + sc, u);
          if (!LOCA_CHECK_SPAN(o2, 16, NB * PT_BK * 2)) continue;
          *reinterpret_cast<uint4*>(sp + PL::b_off + o0) = bh[j];
          *reinterpret_cast<uint4*>(sp + PL::b_off + o1) = bm[j];
          *reinterpret_cast<uint4*>(sp + PL::b_off + o2) = bl[j];
        }
        fence_proxy_async_smem();  // the split tiles visible to the tensor cores
        __syncwarp();
        if (lane == 0) mbar_arrive(split_full(b));
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

template <int KN>
cudaError_t launch_kn(const float* gram, const float* cross, const float* A, int L, int64_t d, int k, float* GA,
                      float* CA, int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  CUtensorMap tmG, tmC, tmA;
  memset(&tmG, 0, sizeof(tmG));
  memset(&tmC, 0, sizeof(tmC));
  memset(&tmA, 0, sizeof(tmA));
  if (!make_map_f32(&tmG, gram, uint64_t(d), uint64_t(d), uint64_t(L), PT_BK, PT_TM, true) ||
      !make_map_f32(&tmC, cross, uint64_t(d), uint64_t(d), uint64_t(L), PT_BK, PT_TM, true) ||
      !make_map_f32(&tmA, A, uint64_t(k), uint64_t(d), uint64_t(L), uint32_t(k), PT_BK, false))
    return cudaErrorInvalidValue;
  PtGeo g;
  g.L = L;
  g.k = k;
  g.d = d;
  g.nrt = int((d + PT_TM - 1) / PT_TM);
  g.nkb = int((d + PT_BK - 1) / PT_BK);
  g.items = L * 2 * g.nrt;
  cudaError_t e = cudaMemsetAsync(abort_flag, 0, sizeof(int32_t), s);
  if (e != cudaSuccess) return e;
  int grid = sm_count();
  if (grid > g.items) grid = g.items;
  const uint32_t shm = PtLayout<KN>::smem_bytes;
  e = cudaFuncSetAttribute(k_project_tc<KN>, cudaFuncAttributeMaxDynamicSharedMemorySize, int(shm));
  if (e != cudaSuccess) return e;
  k_project_tc<KN><<<unsigned(grid), PT_THREADS, shm, s>>>(tmG, tmC, tmA, g, GA, CA, status, abort_flag,
                                                           wait_limit_ns());
  return cudaGetLastError();
}

}  // namespace

bool project_tc_supported(const float* gram, const float* cross, const float* A, int64_t d, int k) {
  auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  return d % 4 == 0 && k % 4 == 0 && k >= 4 && k <= 32 && d < (int64_t(1) << 31) && a16(gram) && a16(cross) &&
         a16(A) && tensor_map_encoder() != nullptr;
}

cudaError_t launch_project_tc(const float* gram, const float* cross, const float* A, int L, int64_t d, int k,
                              float* GA, float* CA, int32_t* status, int32_t* abort_flag, cudaStream_t s) {
  if (k <= 16) return launch_kn<16>(gram, cross, A, L, d, k, GA, CA, status, abort_flag, s);
  return launch_kn<32>(gram, cross, A, L, d, k, GA, CA, status, abort_flag, s);
}

}  // namespace loca
