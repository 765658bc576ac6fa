// Index bounds checks of the LOCA_DEBUG build.
//
// Every kernel guards its global accesses whose index it computes (and the coordinates of its
// TMA stores) with these macros:
//   LOCA_CHECK(i, n)         0 <= i < n
//   LOCA_CHECK_SPAN(i, k, n) the k elements i .. i + k - 1 lie in [0, n)
//   LOCA_REQUIRE(cond)       any other invariant (alignment of a TMA coordinate, a sign)
// The extent n is the one the kernel derives from the sizes of the call (L * N * d for T, ...),
// so a check fails when the index arithmetic leaves the buffer the caller passed.
//
// Built with -DLOCA_DEBUG a macro is an expression that is true when the check holds; when it
// fails it records LOCA_ERR_BOUNDS and the source line in this translation unit's debug word
// (first failure wins), and the caller skips the access.  Nothing traps: the kernel runs on,
// the host reads the word through loca_device_status.  Without LOCA_DEBUG every macro is the
// constant true and the checks compile away.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/loca.h"

namespace loca {

// Copies one translation unit's debug word (code, source line) to the host and clears it.
typedef cudaError_t (*DebugWordReader)(int32_t* code, int32_t* line);

// Adds a reader to the list loca_device_status consults (called by static initialisers of the
// LOCA_DEBUG build); returns true.
bool register_debug_word(DebugWordReader reader, const char* file);

}  // namespace loca

#ifdef LOCA_DEBUG

namespace loca {
namespace {

__device__ int32_t g_debug_word[2];  // first failed check: code, source line

cudaError_t read_debug_word(int32_t* code, int32_t* line) {
  int32_t w[2] = {0, 0};
  cudaError_t e = cudaMemcpyFromSymbol(w, g_debug_word, sizeof(w));
  if (e == cudaSuccess && w[0] != 0) {
    const int32_t zero[2] = {0, 0};
    e = cudaMemcpyToSymbol(g_debug_word, zero, sizeof(zero));
  }
  *code = w[0];
  *line = w[1];
  return e;
}

[[maybe_unused]] const bool g_debug_word_registered = register_debug_word(&read_debug_word, __BASE_FILE__);

__device__ __noinline__ bool debug_fail(int line) {
  if (atomicCAS(&g_debug_word[0], 0, int32_t(LOCA_ERR_BOUNDS)) == 0) atomicExch(&g_debug_word[1], line);
  return false;
}

}  // namespace
}  // namespace loca

#define LOCA_CHECK(i, n) \
  ((int64_t(i) >= 0 && int64_t(i) < int64_t(n)) ? true : ::loca::debug_fail(__LINE__))
#define LOCA_CHECK_SPAN(i, k, n) \
  ((int64_t(i) >= 0 && int64_t(i) + int64_t(k) <= int64_t(n)) ? true : ::loca::debug_fail(__LINE__))
#define LOCA_REQUIRE(cond) ((cond) ? true : ::loca::debug_fail(__LINE__))

#else

#define LOCA_CHECK(i, n) true
#define LOCA_CHECK_SPAN(i, k, n) true
#define LOCA_REQUIRE(cond) true

#endif
