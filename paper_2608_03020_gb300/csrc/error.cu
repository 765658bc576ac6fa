// Top-layer error at the frozen head (Eq. 4; Lemma "Top-layer error", S3).
//
// One warp per logit row.  Each lane streams its share of the row with 16-byte loads and
// keeps a running maximum and a sum of exp(z - max) rescaled whenever the maximum grows,
// so the row is read from HBM exactly once; the 32 partial (max, sum) pairs are merged with
// warp shuffles.  The C label columns are then gathered to form
//   E[n, c] = w_n (exp(z[n, col_c] - lse_n) - [y_n == c]),   ce[n] = w_n (lse_n - z[n, col_{y_n}]).
// The running maximum and sum are kept in base-2 units (t = z log2 e), so each logit costs one
// FMA and one exp2f; lse = (m + log2 s) ln 2.
// Bound: HBM read of the logits (N * V * elsize bytes); for V == C the kernel is launch-bound.
#include <cuda_bf16.h>
#include <math.h>

#include "loca_internal.h"

namespace loca {
namespace {

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(__nv_bfloat16 v) { return __bfloat162float(v); }

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// running maximum m and sum s of 2^(t - m) over t = z log2 e seen so far
struct RunMax {
  float m = -INFINITY;
  float s = 0.f;
  __device__ __forceinline__ void rescale_to(float mn) {
    if (mn > m) {
      s = (m == -INFINITY) ? 0.f : s * exp2f(m - mn);
      m = mn;
    }
  }
  __device__ __forceinline__ void add(float z) {  // one logit (natural units)
    rescale_to(z * kLog2e);
    if (m != -INFINITY) s += exp2f(fmaf(z, kLog2e, -m));
  }
};

__device__ __forceinline__ void merge(RunMax& a, float m2, float s2) {
  const float mn = fmaxf(a.m, m2);
  if (mn == -INFINITY) return;
  const float sa = (a.m == -INFINITY) ? 0.f : a.s * exp2f(a.m - mn);
  const float sb = (m2 == -INFINITY) ? 0.f : s2 * exp2f(m2 - mn);
  a.m = mn;
  a.s = sa + sb;
}

// 16-byte vector of logits converted to fp32.
template <typename Tz>
struct Vec16;
template <>
struct Vec16<float> {
  static constexpr int n = 4;
  __device__ __forceinline__ static void load(const float* p, float* v) {
    const float4 q = __ldg(reinterpret_cast<const float4*>(p));
    v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
  }
};
template <>
struct Vec16<__nv_bfloat16> {
  static constexpr int n = 8;
  __device__ __forceinline__ static void load(const __nv_bfloat16* p, float* v) {
    const uint4 q = __ldg(reinterpret_cast<const uint4*>(p));
    const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      v[2 * i] = __uint_as_float(w[i] << 16);
      v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
};

template <typename Tz>
__device__ __forceinline__ void accumulate_vec(RunMax& a, const float* v) {
  constexpr int n = Vec16<Tz>::n;
  float vm = v[0];
#pragma unroll
  for (int i = 1; i < n; ++i) vm = fmaxf(vm, v[i]);
  a.rescale_to(vm * kLog2e);
  if (a.m == -INFINITY) return;
  float t = 0.f;
#pragma unroll
  for (int i = 0; i < n; ++i) t += exp2f(fmaf(v[i], kLog2e, -a.m));
  a.s += t;
}

template <typename Tz>
__global__ void __launch_bounds__(256) k_head_error(const Tz* __restrict__ z, int64_t N, int64_t V,
                                                    int64_t ldz, const int32_t* __restrict__ cols,
                                                    int C, const int32_t* __restrict__ y,
                                                    const float* __restrict__ w, int normaliser,
                                                    int vec_ok, float* __restrict__ E,
                                                    float* __restrict__ ce) {
  constexpr int VN = Vec16<Tz>::n;
  const int lane = threadIdx.x & 31;
  const int64_t warp0 = (int64_t(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = (int64_t(gridDim.x) * blockDim.x) >> 5;
  for (int64_t n = warp0; n < N; n += nwarps) {
    const Tz* row = z + n * ldz;
    if (!LOCA_CHECK_SPAN(n * ldz, V, (N - 1) * ldz + V)) continue;
    RunMax a0, a1;
    if (normaliser == 0) {
      int64_t j0 = 0;
      if (vec_ok) {
        const int64_t nvec = V / VN;
        int64_t vi = lane;
        // two independent 16-byte loads in flight per lane per iteration
        for (; vi + 32 < nvec; vi += 64) {
          float v0[VN], v1[VN];
          Vec16<Tz>::load(row + vi * VN, v0);
          Vec16<Tz>::load(row + (vi + 32) * VN, v1);
          accumulate_vec<Tz>(a0, v0);
          accumulate_vec<Tz>(a1, v1);
        }
        for (; vi < nvec; vi += 32) {
          float v0[VN];
          Vec16<Tz>::load(row + vi * VN, v0);
          accumulate_vec<Tz>(a0, v0);
        }
        j0 = nvec * VN;
      }
      for (int64_t j = j0 + lane; j < V; j += 32) a1.add(to_f(row[j]));
    } else {
      for (int c = lane; c < C; c += 32) {
        const int32_t col = cols[c];
        if (LOCA_CHECK(col, V)) a0.add(to_f(row[col]));
      }
    }
    merge(a0, a1.m, a1.s);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      const float m2 = __shfl_xor_sync(0xffffffffu, a0.m, off);
      const float s2 = __shfl_xor_sync(0xffffffffu, a0.s, off);
      merge(a0, m2, s2);
    }
    const float lse = (a0.m + log2f(a0.s)) * kLn2;
    const int yn = y[n];
    const float wn = (yn < 0) ? 0.f : (w ? w[n] : 1.f);
    for (int c = lane; c < C; c += 32) {
      const int32_t col = cols[c];
      const float zc = LOCA_CHECK(col, V) ? to_f(row[col]) : 0.f;
      if (LOCA_CHECK(n * C + c, N * C)) E[n * C + c] = wn * (expf(zc - lse) - (c == yn ? 1.f : 0.f));
    }
    if (ce != nullptr && lane == 0 && LOCA_CHECK(n, N)) {
      float cn = 0.f;
      if (yn >= 0 && LOCA_CHECK(yn, C)) {
        const int32_t cy = cols[yn];
        if (LOCA_CHECK(cy, V)) cn = wn * (lse - to_f(row[cy]));
      }
      ce[n] = cn;
    }
  }
}

}  // namespace

cudaError_t launch_head_error(const void* z, int dtype, int64_t N, int64_t V, int64_t ldz,
                              const int32_t* cols, int C, const int32_t* y, const float* w,
                              int normaliser, float* E, float* ce, cudaStream_t s) {
  if (N == 0) return cudaSuccess;
  const int threads = 256;
  int64_t blocks = (N + 7) / 8;
  const int64_t cap = int64_t(sm_count()) * 16;
  if (blocks > cap) blocks = cap;
  const size_t es = dtype == LOCA_BF16 ? 2 : 4;
  const int vec_ok = (reinterpret_cast<uintptr_t>(z) % 16 == 0) && ((ldz * es) % 16 == 0);
  if (dtype == LOCA_BF16) {
    k_head_error<__nv_bfloat16><<<unsigned(blocks), threads, 0, s>>>(
        static_cast<const __nv_bfloat16*>(z), N, V, ldz, cols, C, y, w, normaliser, vec_ok, E, ce);
  } else {
    k_head_error<float><<<unsigned(blocks), threads, 0, s>>>(static_cast<const float*>(z), N, V,
                                                             ldz, cols, C, y, w, normaliser,
                                                             vec_ok, E, ce);
  }
  return cudaGetLastError();
}

}  // namespace loca
