// loca_accumulate_noalloc: loca_accumulate without a caller-provided workspace.
//
// Some callers cannot hand the library a scratch buffer: a host program whose device memory
// is reserved up front by another owner (an inference server or a plugin host that exposes no
// allocator), or a C caller that must not call cudaMalloc on its hot loop because the call
// may synchronise the device and take an unbounded time.  This entry point serves them: its
// scratch lives in a fixed array in the library's own device memory, created when the library
// is loaded and held by every GPU that loads it until the process exits.
//
// The array holds, for up to kNoAllocMaxBlocks blocks, the per-thread-block partial sums of
// ||X_l||^2, the step alpha_l, and the launch-local flag of the tensor-core kernel's bounded
// waits.  Every call reuses the same array and leaves the previous call's values in it; the
// partial sums and alpha are overwritten before they are read, and the flag is cleared by the
// launch.  Two calls whose work overlaps on the GPU (different streams, or different host
// threads without ordering) race on the array and produce wrong results: order them.
#include <cuda_runtime.h>

#include <mutex>

#include "loca_internal.h"

// Largest number of blocks one call may pass, and the layout of the scratch array:
// partial sums (one row of 1024 doubles per block), alpha (one float per block), wait flag.
constexpr int kNoAllocMaxBlocks = 64;
constexpr size_t kPartialBytes = size_t(kNoAllocMaxBlocks) * 1024 * sizeof(double);  // 512 KiB
constexpr size_t kAlphaBytes = 256;  // kNoAllocMaxBlocks floats
constexpr size_t kFlagBytes = 256;
constexpr size_t kScratchBytes = kPartialBytes + kAlphaBytes + kFlagBytes;  // 524,800 bytes

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

namespace loca {
namespace {

constexpr int kMaxDevices = 64;

bool na_aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Device address of the scratch array on the current device.  The array's name in host code
// is only a host-side handle, so the address is looked up with cudaGetSymbolAddress, once per
// device, with that device current.
unsigned char* scratch_on_current_device(cudaError_t* err) {
  static unsigned char* cache[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  *err = cudaGetDevice(&dev);
  if (*err != cudaSuccess) return nullptr;
  if (dev < 0 || dev >= kMaxDevices) {
    *err = cudaErrorInvalidDevice;
    return nullptr;
  }
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == nullptr) {
    void* p = nullptr;
    *err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (*err != cudaSuccess) return nullptr;
    cache[dev] = static_cast<unsigned char*>(p);
  }
  return cache[dev];
}

}  // namespace
}  // namespace loca

using namespace loca;

extern "C" int loca_accumulate_noalloc(const void* X, const void* T, int dtype, int32_t L, int64_t N,
                                       int64_t d, const double* tsq, float eta, int zero_first,
                                       float* gram, float* cross, double* xsq_total, void* stream) {
  set_error_message(LOCA_OK, "");
  if (L < 1 || L > kNoAllocMaxBlocks)
    return set_error_message(LOCA_ERR_SHAPE,
                   "loca_accumulate_noalloc handles 1 <= L <= %d blocks (its fixed scratch is sized "
                   "for %d); got L=%d: use loca_accumulate with a workspace",
                   kNoAllocMaxBlocks, kNoAllocMaxBlocks, L);
  if (N < 0 || d < 1) return set_error_message(LOCA_ERR_SHAPE, "need N >= 0 and d >= 1");
  if (dtype != LOCA_F32 && dtype != LOCA_BF16)
    return set_error_message(LOCA_ERR_UNSUPPORTED_DTYPE, "dtype must be LOCA_F32 or LOCA_BF16");
  if (!(eta >= 0.f)) return set_error_message(LOCA_ERR_INVALID_ARG, "eta must be >= 0");
  if (!tsq || !gram || !cross || !xsq_total || (N > 0 && (!X || !T)))
    return set_error_message(LOCA_ERR_INVALID_ARG, "X, T, tsq, gram, cross and xsq_total are required");
  if (!na_aligned(gram, 16) || !na_aligned(cross, 16) || !na_aligned(tsq, 8) || !na_aligned(xsq_total, 8))
    return set_error_message(LOCA_ERR_ALIGNMENT, "gram and cross need 16-byte, tsq and xsq_total 8-byte alignment");
  if (dtype == LOCA_BF16) {
    if (d % 8 != 0) return set_error_message(LOCA_ERR_SHAPE, "the bf16 path needs d %% 8 == 0, got d=%lld", (long long)d);
    if (d > 65536 || N > 2147483647LL) return set_error_message(LOCA_ERR_SHAPE, "the bf16 path needs d <= 65536 and N < 2^31");
    if (N > 0 && (!na_aligned(X, 16) || !na_aligned(T, 16)))
      return set_error_message(LOCA_ERR_ALIGNMENT, "the bf16 path needs 16-byte aligned X and T");
  } else if (N > 0 && (!na_aligned(X, 4) || !na_aligned(T, 4))) {
    return set_error_message(LOCA_ERR_ALIGNMENT, "X and T need 4-byte alignment");
  }
  cudaError_t e = cudaSuccess;
  unsigned char* scratch = scratch_on_current_device(&e);
  if (scratch == nullptr)
    return set_error_message(LOCA_ERR_CUDA, "cannot resolve the scratch array's device address: %s", cudaGetErrorString(e));
  double* partials = reinterpret_cast<double*>(scratch);
  float* alpha = reinterpret_cast<float*>(scratch + kPartialBytes);
  int32_t* abort_flag = reinterpret_cast<int32_t*>(scratch + kPartialBytes + kAlphaBytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  e = launch_sumsq_and_step(X, dtype, L, N, d, tsq, eta, zero_first, xsq_total, partials, alpha, s);
  if (e != cudaSuccess) return set_error_message(LOCA_ERR_CUDA, "sum of squares: %s", cudaGetErrorString(e));
  if (N == 0) {
    if (zero_first) {
      e = cudaMemsetAsync(gram, 0, sizeof(float) * size_t(L) * size_t(d) * size_t(d), s);
      if (e == cudaSuccess) e = cudaMemsetAsync(cross, 0, sizeof(float) * size_t(L) * size_t(d) * size_t(d), s);
      if (e != cudaSuccess) return set_error_message(LOCA_ERR_CUDA, "zeroing: %s", cudaGetErrorString(e));
    }
    return LOCA_OK;
  }
  if (dtype == LOCA_BF16) {
    int32_t* status = device_status_word();
    if (!status) return set_error_message(LOCA_ERR_CUDA, "cannot resolve the device status word");
    e = launch_gram_cross_tc(X, T, L, N, d, alpha, zero_first, gram, cross, status, abort_flag, s);
  } else {
    e = launch_gram_cross_f32(static_cast<const float*>(X), static_cast<const float*>(T), L, N, d, alpha,
                              zero_first, gram, cross, s);
  }
  if (e != cudaSuccess) return set_error_message(LOCA_ERR_CUDA, "Gram/cross launch: %s", cudaGetErrorString(e));
  return LOCA_OK;
}
