// Host memory for inputs that stream to the GPU (loca_host_alloc / loca_host_free).
//
// Host-to-device copies read page-locked host memory through the GPU's address translation.
// With 4 KiB pages a buffer of tens of GB copies at a rate that varies from run to run (91 to
// 211 GB/s measured for 26 GB of bf16 activations on one GB300 machine); backed by 2 MiB pages it
// copies at the link rate every time (211-212 GB/s).  So the buffer is an anonymous mapping,
// 2 MiB aligned, advised to use transparent huge pages, touched once (in parallel) so that the
// pages exist before CUDA registers them, and then registered (page-locked, device-visible).
#include <cuda_runtime.h>
#include <sys/mman.h>

#include <cstdint>
#include <cstring>
#include <map>
#include <mutex>
#include <thread>
#include <vector>

#include "loca_internal.h"

namespace {

constexpr size_t kHuge = size_t(2) << 20;

struct Mapping {
  void* base;
  size_t len;
};
std::mutex g_mu;
std::map<void*, Mapping>& registry() {
  static std::map<void*, Mapping> m;
  return m;
}

void parallel_zero(char* p, size_t n) {
  unsigned nt = std::thread::hardware_concurrency();
  if (nt == 0) nt = 1;
  if (nt > 32) nt = 32;
  if (n < (size_t(64) << 20)) nt = 1;
  const size_t chunk = ((n + nt - 1) / nt + kHuge - 1) / kHuge * kHuge;
  std::vector<std::thread> th;
  for (unsigned t = 0; t < nt; ++t) {
    const size_t a = size_t(t) * chunk;
    if (a >= n) break;
    const size_t b = (a + chunk < n) ? a + chunk : n;
    th.emplace_back([p, a, b] { memset(p + a, 0, b - a); });
  }
  for (auto& t : th) t.join();
}

}  // namespace

extern "C" {

int loca_host_alloc(size_t bytes, void** ptr) {
  if (!ptr) return loca::set_error_message(LOCA_ERR_INVALID_ARG, "ptr is NULL");
  *ptr = nullptr;
  if (bytes == 0) return LOCA_OK;
  const size_t len = (bytes + kHuge - 1) / kHuge * kHuge;
  void* raw = mmap(nullptr, len + kHuge, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == MAP_FAILED) return loca::set_error_message(LOCA_ERR_INVALID_ARG, "mmap of %zu bytes failed", len + kHuge);
  char* p = reinterpret_cast<char*>((reinterpret_cast<uintptr_t>(raw) + kHuge - 1) & ~uintptr_t(kHuge - 1));
  madvise(p, len, MADV_HUGEPAGE);  // a hint: without huge pages the buffer still works
  parallel_zero(p, len);
  const cudaError_t e = cudaHostRegister(p, len, cudaHostRegisterDefault);
  if (e != cudaSuccess) {
    munmap(raw, len + kHuge);
    return loca::set_error_message(LOCA_ERR_CUDA, "cudaHostRegister of %zu bytes: %s", len, cudaGetErrorString(e));
  }
  {
    std::lock_guard<std::mutex> lock(g_mu);
    registry()[p] = Mapping{raw, len + kHuge};
  }
  *ptr = p;
  return LOCA_OK;
}

int loca_host_free(void* ptr) {
  if (!ptr) return LOCA_OK;
  Mapping m{};
  {
    std::lock_guard<std::mutex> lock(g_mu);
    auto it = registry().find(ptr);
    if (it == registry().end())
      return loca::set_error_message(LOCA_ERR_INVALID_ARG, "pointer was not returned by loca_host_alloc");
    m = it->second;
    registry().erase(it);
  }
  const cudaError_t e = cudaHostUnregister(ptr);
  munmap(m.base, m.len);
  if (e != cudaSuccess) return loca::set_error_message(LOCA_ERR_CUDA, "cudaHostUnregister: %s", cudaGetErrorString(e));
  return LOCA_OK;
}

}  // extern "C"
