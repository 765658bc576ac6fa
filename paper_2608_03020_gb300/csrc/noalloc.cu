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

// Device address of the scratch array in the current context.  The array's name in host code is
// only a host-side handle, so the address is looked up with cudaGetSymbolAddress, with the
// caller's device current, at every call: the lookup allocates nothing, and an address kept from
// an earlier call would outlive the context it belongs to (cudaDeviceReset creates a new one).
unsigned char* scratch_on_current_device(cudaError_t* err) {
  void* p = nullptr;
  *err = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  return *err == cudaSuccess ? static_cast<unsigned char*>(p) : nullptr;
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
  // the same checks as loca_accumulate
  const int rc = validate_accumulate(X, T, dtype, L, N, d, tsq, eta, gram, cross, xsq_total);
  if (rc != LOCA_OK) return rc;
  cudaError_t e = cudaSuccess;
  unsigned char* scratch = scratch_on_current_device(&e);
  if (scratch == nullptr)
    return set_error_message(LOCA_ERR_CUDA, "cannot resolve the scratch array's device address: %s", cudaGetErrorString(e));
  double* partials = reinterpret_cast<double*>(scratch);
  float* alpha = reinterpret_cast<float*>(scratch + kPartialBytes);
  int32_t* abort_flag = reinterpret_cast<int32_t*>(scratch + kPartialBytes + kAlphaBytes);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the same launches as loca_accumulate, with the scratch array in place of the workspace
  const int rs = run_batch_step(X, dtype, L, N, d, tsq, eta, zero_first, xsq_total, alpha, partials, s);
  if (rs != LOCA_OK) return rs;
  return run_gram_cross(X, T, dtype, L, N, d, alpha, zero_first, gram, cross, abort_flag, s);
}
