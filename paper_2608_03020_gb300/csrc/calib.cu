// One-shot reduced-rank feedback fit (Eq. 5; S5) — kernels follow.
#include "loca_internal.h"

namespace loca {

size_t calib_workspace_bytes(int64_t, int, int64_t, int, int) { return 0; }

cudaError_t launch_calib_fit(const float*, const float*, int64_t, int, int64_t, int, float, int,
                             float*, float*, float*, void*, cudaStream_t) {
  return cudaErrorNotSupported;
}

}  // namespace loca
