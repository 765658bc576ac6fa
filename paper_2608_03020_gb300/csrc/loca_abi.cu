// C ABI entry points: host-side validation, workspace layout, and dispatch to the kernels.
// See include/loca.h for the contract of each function.
#include <cuda_runtime.h>

#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <atomic>
#include <mutex>
#include <vector>

#include "loca_internal.h"

namespace loca {
namespace {

thread_local char g_msg[512] = "";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* where) {
  return fail(LOCA_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

__device__ int32_t g_status_word = 0;

constexpr int kMaxDevices = 64;

}  // namespace

TensorMapEncodeFn tensor_map_encoder() {
  static TensorMapEncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<TensorMapEncodeFn>(p);
  });
  return fn;
}

int set_error_message(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
  va_end(ap);
  return code;
}

int sm_count() {
  static int cache[kMaxDevices] = {};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return 148;
  if (cache[dev] == 0) {
    int v = 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || v <= 0)
      v = 148;
    cache[dev] = v;
  }
  return cache[dev];
}

namespace {
std::atomic<unsigned long long> g_wait_limit_ns{0};
}

unsigned long long wait_limit_ns() {
  const unsigned long long v = g_wait_limit_ns.load(std::memory_order_relaxed);
  return v == 0 ? 4000000000ull : v;
}

namespace {
struct DebugWord {
  DebugWordReader read;
  const char* file;
};
struct DebugWords {
  std::mutex mu;
  std::vector<DebugWord> list;  // filled by static initialisers, before any entry point runs
};
DebugWords& debug_words() {
  static DebugWords w;
  return w;
}
}  // namespace

bool register_debug_word(DebugWordReader reader, const char* file) {
  DebugWords& w = debug_words();
  std::lock_guard<std::mutex> lock(w.mu);
  w.list.push_back(DebugWord{reader, file});
  return true;
}

int32_t* device_status_word() {
  static int32_t* cache[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (cache[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    cache[dev] = static_cast<int32_t*>(p);
  }
  return cache[dev];
}

}  // namespace loca

using namespace loca;

namespace {

// ---- workspace layouts (offsets are 256-byte aligned)
struct TargetsWs {
  size_t partials, total;
};
TargetsWs targets_ws(int64_t N, int32_t L, int64_t d) {
  TargetsWs w{};
  w.partials = 0;
  w.total = targets_workspace_bytes(N, L, d);
  return w;
}

struct AccumWs {
  size_t partials, alpha, abort_flag, total;
};
AccumWs accum_ws(int32_t L) {
  AccumWs w{};
  w.partials = 0;
  w.alpha = align256(sizeof(double) * size_t(L) * size_t(sumsq_num_partials()));
  w.abort_flag = w.alpha + align256(sizeof(float) * size_t(L));
  w.total = w.abort_flag + 256;
  return w;
}

struct SolveWs {
  size_t ga, ca, fac, arec, flag, total;
};
SolveWs solve_ws(int32_t L, int64_t d, int32_t k) {
  SolveWs w{};
  const size_t one = align256(sizeof(float) * size_t(project_split()) * size_t(L) * size_t(d) * size_t(k));
  w.ga = 0;
  w.ca = one;
  w.fac = 2 * one;  // per-candidate Cholesky factors
  w.arec = w.fac + align256(chol_workspace_bytes(L));  // A's split slabs for the tensor-core projection
  w.flag = w.arec + align256(project_tc_workspace_bytes(L, d, k));  // abort flag of its waits
  w.total = w.flag + 256;
  return w;
}

int check_ws(void* ws, size_t have, size_t need) {
  if (need == 0) return LOCA_OK;
  if (ws == nullptr) return fail(LOCA_ERR_WORKSPACE, "workspace is NULL but %zu bytes are required", need);
  if (have < need)
    return fail(LOCA_ERR_WORKSPACE, "workspace of %zu bytes is smaller than the %zu required", have, need);
  if (!aligned(ws, 256)) return fail(LOCA_ERR_ALIGNMENT, "workspace must be 256-byte aligned");
  return LOCA_OK;
}

char* ws_at(void* ws, size_t off) { return static_cast<char*>(ws) + off; }

// Per-device copy stream and events of loca_accumulate_streamed: copied[s] marks the end of the
// latest copy into staging slot s, consumed[s] the end of the kernels that last read slot s.
struct CopyLane {
  cudaStream_t copy = nullptr;
  cudaEvent_t copied[2] = {nullptr, nullptr};
  cudaEvent_t consumed[2] = {nullptr, nullptr};
  std::mutex mu;  // one call enqueues its copy / wait / record sequence at a time
};

CopyLane* copy_lane() {
  static CopyLane* lanes[kMaxDevices] = {};
  static std::mutex mu;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return nullptr;
  std::lock_guard<std::mutex> lock(mu);
  if (lanes[dev] == nullptr) {
    CopyLane* c = new CopyLane();
    cudaError_t e = cudaStreamCreateWithFlags(&c->copy, cudaStreamNonBlocking);
    for (int i = 0; i < 2 && e == cudaSuccess; ++i) {
      e = cudaEventCreateWithFlags(&c->copied[i], cudaEventDisableTiming);
      if (e == cudaSuccess) e = cudaEventCreateWithFlags(&c->consumed[i], cudaEventDisableTiming);
    }
    if (e != cudaSuccess) {
      for (int i = 0; i < 2; ++i) {
        if (c->copied[i]) cudaEventDestroy(c->copied[i]);
        if (c->consumed[i]) cudaEventDestroy(c->consumed[i]);
      }
      if (c->copy) cudaStreamDestroy(c->copy);
      delete c;
      fail(LOCA_ERR_CUDA, "cannot create the copy stream and events: %s", cudaGetErrorString(e));
      return nullptr;
    }
    lanes[dev] = c;
  }
  return lanes[dev];
}

}  // namespace

extern "C" {

int loca_version(void) { return 100; }

const char* loca_last_error_string(void) { return g_msg; }

int loca_set_wait_limit(uint64_t ns) {
  g_wait_limit_ns.store(ns, std::memory_order_relaxed);
  return LOCA_OK;
}

int loca_device_status(int32_t* host_status, void* stream) {
  if (host_status == nullptr) return fail(LOCA_ERR_INVALID_ARG, "host_status is NULL");
  int32_t* w = device_status_word();
  if (w == nullptr) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemcpyAsync(host_status, w, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
  if (e == cudaSuccess) e = cudaMemsetAsync(w, 0, sizeof(int32_t), s);
  if (e == cudaSuccess) e = cudaStreamSynchronize(s);
  if (e != cudaSuccess) return cuda_fail(e, "loca_device_status");
  // debug build: the first failed bounds check of each translation unit (all words are cleared)
  for (const DebugWord& dw : debug_words().list) {
    int32_t code = 0, line = 0;
    e = dw.read(&code, &line);
    if (e != cudaSuccess) return cuda_fail(e, "loca_device_status (debug word)");
    if (code != 0 && *host_status == LOCA_OK) {
      *host_status = code;
      set_error_message(code, "device: index outside its buffer at %s:%d", dw.file, int(line));
    }
  }
  return LOCA_OK;
}

int loca_debug_build(void) {
#ifdef LOCA_DEBUG
  return 1;
#else
  return 0;
#endif
}

int loca_error(const void* logits, int logit_dtype, int64_t N, int64_t V, int64_t ldz,
               const int32_t* label_cols, int32_t C, const int32_t* y, const float* w,
               int normaliser, float* E, float* ce, void* stream) {
  g_msg[0] = 0;
  if (N < 0 || V < 1 || ldz < V) return fail(LOCA_ERR_SHAPE, "need N >= 0, V >= 1, ldz >= V (N=%lld V=%lld ldz=%lld)", (long long)N, (long long)V, (long long)ldz);
  if (C < 1 || C > 1024 || C > V) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= min(V, 1024), got C=%d", C);
  if (logit_dtype != LOCA_F32 && logit_dtype != LOCA_BF16)
    return fail(LOCA_ERR_UNSUPPORTED_DTYPE, "logit_dtype must be LOCA_F32 or LOCA_BF16");
  if (normaliser != 0 && normaliser != 1) return fail(LOCA_ERR_INVALID_ARG, "normaliser must be 0 or 1");
  if (N == 0) return LOCA_OK;
  if (!logits || !label_cols || !y || !E) return fail(LOCA_ERR_INVALID_ARG, "logits, label_cols, y and E are required");
  const size_t es = logit_dtype == LOCA_BF16 ? 2 : 4;
  if (!aligned(logits, es) || !aligned(label_cols, 4) || !aligned(y, 4) || !aligned(E, 4) ||
      (w && !aligned(w, 4)) || (ce && !aligned(ce, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be aligned to their element size");
  cudaError_t e = launch_head_error(logits, logit_dtype, N, V, ldz, label_cols, C, y, w, normaliser,
                                    E, ce, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_error launch");
  return LOCA_OK;
}

int loca_targets_workspace_size(int64_t N, int32_t L, int64_t d, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (N < 0 || L < 1 || d < 1) return fail(LOCA_ERR_SHAPE, "need N >= 0, L >= 1, d >= 1");
  *bytes = targets_ws(N, L, d).total;
  return LOCA_OK;
}

int loca_targets(const float* E, int64_t N, int32_t C, const float* P, const float* Q, int32_t L,
                 int32_t r, int64_t d, void* T, int t_dtype, double* tsq, void* workspace,
                 size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (N < 0 || L < 1 || L > 65535 || d < 1) return fail(LOCA_ERR_SHAPE, "need N >= 0, 1 <= L <= 65535, d >= 1");
  if (C < 1 || C > targets_max_C()) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= %d, got C=%d", targets_max_C(), C);
  if (r < 1 || r > targets_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got %d", targets_max_r(), r);
  if (t_dtype != LOCA_F32 && t_dtype != LOCA_BF16)
    return fail(LOCA_ERR_UNSUPPORTED_DTYPE, "t_dtype must be LOCA_F32 or LOCA_BF16");
  if ((N > 0 && (!E || !T)) || !P || !Q) return fail(LOCA_ERR_INVALID_ARG, "E, P, Q and T are required");
  const size_t es = t_dtype == LOCA_BF16 ? 2 : 4;
  if (!aligned(E, 4) || !aligned(P, 4) || !aligned(Q, 4) || !aligned(T, 16) || (tsq && !aligned(tsq, 8)))
    return fail(LOCA_ERR_ALIGNMENT, "E, P, Q need 4-byte, T 16-byte and tsq 8-byte alignment");
  (void)es;
  const int rc = check_ws(workspace, workspace_bytes, targets_ws(N, L, d).total);
  if (rc != LOCA_OK) return rc;
  int32_t* status = device_status_word();
  if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  cudaError_t e = launch_targets(E, N, C, P, Q, L, r, d, T, t_dtype, tsq, workspace, status,
                                 static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_targets launch");
  return LOCA_OK;
}

}  // extern "C"

namespace loca {

int validate_stats_inputs(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                          bool need_T) {
  if (L < 1 || L > 255 || N < 0 || d < 1) return fail(LOCA_ERR_SHAPE, "need 1 <= L <= 255, N >= 0, d >= 1");
  if (dtype != LOCA_F32 && dtype != LOCA_BF16)
    return fail(LOCA_ERR_UNSUPPORTED_DTYPE, "dtype must be LOCA_F32 or LOCA_BF16");
  if (N > 0 && (!X || (need_T && !T))) return fail(LOCA_ERR_INVALID_ARG, "X and T are required");
  if (dtype == LOCA_BF16) {
    if (d % 8 != 0) return fail(LOCA_ERR_SHAPE, "the bf16 path needs d %% 8 == 0 (16-byte rows), got d=%lld", (long long)d);
    if (d > 65536 || N > 2147483647LL) return fail(LOCA_ERR_SHAPE, "the bf16 path needs d <= 65536 and N < 2^31");
    if (N > 0 && (!aligned(X, 16) || (need_T && !aligned(T, 16))))
      return fail(LOCA_ERR_ALIGNMENT, "the bf16 path needs 16-byte aligned X and T");
  } else {
    if (N > 0 && (!aligned(X, 4) || (need_T && !aligned(T, 4)))) return fail(LOCA_ERR_ALIGNMENT, "X and T need 4-byte alignment");
  }
  return LOCA_OK;
}

int validate_accumulate(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                        const double* tsq, float eta, const float* gram, const float* cross,
                        const double* xsq_total) {
  const int rc = validate_stats_inputs(X, T, dtype, L, N, d, true);
  if (rc != LOCA_OK) return rc;
  if (!(eta >= 0.f)) return fail(LOCA_ERR_INVALID_ARG, "eta must be >= 0");
  if (!tsq || !gram || !cross || !xsq_total)
    return fail(LOCA_ERR_INVALID_ARG, "tsq, gram, cross and xsq_total are required");
  if (!aligned(gram, 16) || !aligned(cross, 16) || !aligned(tsq, 8) || !aligned(xsq_total, 8))
    return fail(LOCA_ERR_ALIGNMENT, "gram and cross need 16-byte, tsq and xsq_total 8-byte alignment");
  return LOCA_OK;
}

int run_batch_step(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const double* tsq,
                   float eta, int zero_first, double* xsq_total, float* alpha, double* partials,
                   cudaStream_t s) {
  cudaError_t e = launch_sumsq_and_step(X, dtype, L, N, d, tsq, eta, zero_first, xsq_total, partials, alpha, s);
  if (e != cudaSuccess) return cuda_fail(e, "batch step: sum of squares");
  return LOCA_OK;
}

int run_gram_cross(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                   const float* alpha, int zero_first, float* gram, float* cross, int32_t* abort_flag,
                   cudaStream_t s) {
  cudaError_t e = cudaSuccess;
  if (N == 0) {
    if (zero_first) {
      e = cudaMemsetAsync(gram, 0, sizeof(float) * size_t(L) * size_t(d) * size_t(d), s);
      if (e == cudaSuccess) e = cudaMemsetAsync(cross, 0, sizeof(float) * size_t(L) * size_t(d) * size_t(d), s);
      if (e != cudaSuccess) return cuda_fail(e, "Gram/cross: zeroing");
    }
    return LOCA_OK;
  }
  if (dtype == LOCA_BF16) {
    int32_t* status = device_status_word();
    if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
    e = launch_gram_cross_tc(X, T, L, N, d, alpha, zero_first, gram, cross, status, abort_flag, s);
  } else {
    e = launch_gram_cross_f32(static_cast<const float*>(X), static_cast<const float*>(T), L, N, d,
                              alpha, zero_first, gram, cross, s);
  }
  if (e != cudaSuccess) return cuda_fail(e, "Gram/cross launch");
  return LOCA_OK;
}

}  // namespace loca

namespace {

size_t batch_step_ws(int32_t L) { return align256(sizeof(double) * size_t(L) * size_t(sumsq_num_partials())); }
constexpr size_t kGramCrossWs = 256;

}  // namespace

extern "C" {

int loca_batch_step_workspace_size(int32_t L, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (L < 1) return fail(LOCA_ERR_SHAPE, "need L >= 1");
  *bytes = batch_step_ws(L);
  return LOCA_OK;
}

int loca_batch_step(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const double* tsq,
                    float eta, int zero_first, double* xsq_total, float* alpha, void* workspace,
                    size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  int rc = validate_stats_inputs(X, nullptr, dtype, L, N, d, false);
  if (rc != LOCA_OK) return rc;
  if (!(eta >= 0.f)) return fail(LOCA_ERR_INVALID_ARG, "eta must be >= 0");
  if (!tsq || !xsq_total || !alpha) return fail(LOCA_ERR_INVALID_ARG, "tsq, xsq_total and alpha are required");
  if (!aligned(tsq, 8) || !aligned(xsq_total, 8) || !aligned(alpha, 4))
    return fail(LOCA_ERR_ALIGNMENT, "tsq and xsq_total need 8-byte, alpha 4-byte alignment");
  rc = check_ws(workspace, workspace_bytes, batch_step_ws(L));
  if (rc != LOCA_OK) return rc;
  return run_batch_step(X, dtype, L, N, d, tsq, eta, zero_first, xsq_total, alpha,
                        reinterpret_cast<double*>(workspace), static_cast<cudaStream_t>(stream));
}

int loca_gram_cross_workspace_size(size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  *bytes = kGramCrossWs;
  return LOCA_OK;
}

int loca_gram_cross(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                    const float* alpha, int zero_first, float* gram, float* cross, void* workspace,
                    size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  int rc = validate_stats_inputs(X, T, dtype, L, N, d, true);
  if (rc != LOCA_OK) return rc;
  if (!alpha || !gram || !cross) return fail(LOCA_ERR_INVALID_ARG, "alpha, gram and cross are required");
  if (!aligned(gram, 16) || !aligned(cross, 16) || !aligned(alpha, 4))
    return fail(LOCA_ERR_ALIGNMENT, "gram and cross need 16-byte, alpha 4-byte alignment");
  rc = check_ws(workspace, workspace_bytes, kGramCrossWs);
  if (rc != LOCA_OK) return rc;
  return run_gram_cross(X, T, dtype, L, N, d, alpha, zero_first, gram, cross,
                        reinterpret_cast<int32_t*>(workspace), static_cast<cudaStream_t>(stream));
}

int loca_targets_sq_workspace_size(int64_t N, int32_t C, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (N < 0 || C < 1 || C > tsq_max_C()) return fail(LOCA_ERR_SHAPE, "need N >= 0 and 1 <= C <= %d", tsq_max_C());
  *bytes = tsq_workspace_bytes(N, C);
  return LOCA_OK;
}

int loca_targets_sq(const float* E, int64_t N, int32_t C, const float* P, const float* Q, int32_t L, int32_t r,
                    int64_t d, double* tsq, void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (N < 0 || L < 1 || L > 65535 || d < 1) return fail(LOCA_ERR_SHAPE, "need N >= 0, 1 <= L <= 65535, d >= 1");
  if (C < 1 || C > tsq_max_C()) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= %d, got C=%d", tsq_max_C(), C);
  if (r < 1 || r > tsq_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got %d", tsq_max_r(), r);
  if ((N > 0 && !E) || !P || !Q || !tsq) return fail(LOCA_ERR_INVALID_ARG, "E, P, Q and tsq are required");
  if (!aligned(E, 4) || !aligned(P, 4) || !aligned(Q, 4) || !aligned(tsq, 8))
    return fail(LOCA_ERR_ALIGNMENT, "E, P, Q need 4-byte and tsq 8-byte alignment");
  const int rc = check_ws(workspace, workspace_bytes, tsq_workspace_bytes(N, C));
  if (rc != LOCA_OK) return rc;
  const cudaError_t e = launch_targets_sq(E, N, C, P, Q, L, r, d, tsq, workspace, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_targets_sq launch");
  return LOCA_OK;
}

int loca_gram_cross_fused_workspace_size(int32_t L, int64_t N, int32_t r, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (L < 1 || N < 0 || r < 1 || r > gram_fused_max_r())
    return fail(LOCA_ERR_SHAPE, "need L >= 1, N >= 0 and 1 <= r <= %d", gram_fused_max_r());
  *bytes = gram_fused_workspace_bytes(L, N, r);
  return LOCA_OK;
}

int loca_gram_cross_fused(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const float* E, int32_t C,
                          const float* P, const float* Q, int32_t r, const float* alpha, int zero_first,
                          float* gram, float* cross, void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (dtype != LOCA_BF16)
    return fail(LOCA_ERR_UNSUPPORTED_DTYPE, "loca_gram_cross_fused takes bf16 X (LOCA_BF16) only");
  int rc = validate_stats_inputs(X, X, dtype, L, N, d, false);
  if (rc != LOCA_OK) return rc;
  if (C < 1 || C > tsq_max_C()) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= %d, got C=%d", tsq_max_C(), C);
  if (r < 1 || r > gram_fused_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got %d", gram_fused_max_r(), r);
  if ((N > 0 && !E) || !P || !Q || !alpha || !gram || !cross)
    return fail(LOCA_ERR_INVALID_ARG, "E, P, Q, alpha, gram and cross are required");
  if (!aligned(gram, 16) || !aligned(cross, 16) || !aligned(alpha, 4) || !aligned(E, 4) || !aligned(P, 4) ||
      !aligned(Q, 4))
    return fail(LOCA_ERR_ALIGNMENT, "gram and cross need 16-byte, alpha, E, P, Q 4-byte alignment");
  rc = check_ws(workspace, workspace_bytes, gram_fused_workspace_bytes(L, N, r));
  if (rc != LOCA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (N == 0) return run_gram_cross(X, X, dtype, L, N, d, alpha, zero_first, gram, cross, nullptr, s);
  int32_t* status = device_status_word();
  if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  const cudaError_t e = launch_gram_cross_fused_tc(X, E, C, P, Q, r, L, N, d, alpha, zero_first, gram, cross, status,
                                                   workspace, s);
  if (e != cudaSuccess) return cuda_fail(e, "loca_gram_cross_fused launch");
  return LOCA_OK;
}

int loca_accumulate_workspace_size(int32_t L, int64_t N, int64_t d, int dtype, size_t* bytes) {
  (void)N;
  (void)d;
  (void)dtype;
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (L < 1) return fail(LOCA_ERR_SHAPE, "need L >= 1");
  *bytes = accum_ws(L).total;
  return LOCA_OK;
}

int loca_accumulate(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                    const double* tsq, float eta, int zero_first, float* gram, float* cross,
                    double* xsq_total, void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  int rc = validate_accumulate(X, T, dtype, L, N, d, tsq, eta, gram, cross, xsq_total);
  if (rc != LOCA_OK) return rc;
  const AccumWs lay = accum_ws(L);
  rc = check_ws(workspace, workspace_bytes, lay.total);
  if (rc != LOCA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* alpha = reinterpret_cast<float*>(ws_at(workspace, lay.alpha));
  rc = run_batch_step(X, dtype, L, N, d, tsq, eta, zero_first, xsq_total, alpha,
                      reinterpret_cast<double*>(ws_at(workspace, lay.partials)), s);
  if (rc != LOCA_OK) return rc;
  return run_gram_cross(X, T, dtype, L, N, d, alpha, zero_first, gram, cross,
                        reinterpret_cast<int32_t*>(ws_at(workspace, lay.abort_flag)), s);
}

int loca_accumulate_streamed(const void* X_host, void* staging, const void* T, int dtype, int32_t L,
                             int64_t N, int64_t d, int32_t group, const double* tsq, float eta,
                             int zero_first, float* gram, float* cross, double* xsq_total,
                             void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  int rc = validate_stats_inputs(staging, T, dtype, L, N, d, true);
  if (rc != LOCA_OK) return rc;
  if (N > 0 && !X_host) return fail(LOCA_ERR_INVALID_ARG, "X_host is required");
  if (group < 1) return fail(LOCA_ERR_SHAPE, "need group >= 1, got %d", group);
  if (group > L) group = L;
  if (!(eta >= 0.f)) return fail(LOCA_ERR_INVALID_ARG, "eta must be >= 0");
  if (!tsq || !gram || !cross || !xsq_total)
    return fail(LOCA_ERR_INVALID_ARG, "tsq, gram, cross and xsq_total are required");
  if (!aligned(gram, 16) || !aligned(cross, 16) || !aligned(tsq, 8) || !aligned(xsq_total, 8))
    return fail(LOCA_ERR_ALIGNMENT, "gram and cross need 16-byte, tsq and xsq_total 8-byte alignment");
  const AccumWs lay = accum_ws(L);
  rc = check_ws(workspace, workspace_bytes, lay.total);
  if (rc != LOCA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* alpha = reinterpret_cast<float*>(ws_at(workspace, lay.alpha));
  double* partials = reinterpret_cast<double*>(ws_at(workspace, lay.partials));
  int32_t* flags = reinterpret_cast<int32_t*>(ws_at(workspace, lay.abort_flag));
  if (N == 0)  // nothing to copy: the statistics of an empty batch
    return loca_accumulate(staging, T, dtype, L, N, d, tsq, eta, zero_first, gram, cross, xsq_total,
                           workspace, workspace_bytes, stream);
  CopyLane* lane = copy_lane();
  if (!lane) return LOCA_ERR_CUDA;  // message set by copy_lane
  std::lock_guard<std::mutex> lock(lane->mu);
  const size_t es = dtype == LOCA_BF16 ? 2 : 4;
  const size_t block_bytes = size_t(N) * size_t(d) * es;
  const size_t dd = size_t(d) * size_t(d);
  for (int32_t l0 = 0, g = 0; l0 < L; l0 += group, ++g) {
    const int32_t nb = (L - l0 < group) ? L - l0 : group;
    const int slot = g & 1;
    char* dst = static_cast<char*>(staging) + size_t(slot) * size_t(group) * block_bytes;
    const char* src = static_cast<const char*>(X_host) + size_t(l0) * block_bytes;
    cudaError_t e = cudaStreamWaitEvent(lane->copy, lane->consumed[slot], 0);
    if (e == cudaSuccess) e = cudaMemcpyAsync(dst, src, size_t(nb) * block_bytes, cudaMemcpyHostToDevice, lane->copy);
    if (e == cudaSuccess) e = cudaEventRecord(lane->copied[slot], lane->copy);
    if (e == cudaSuccess) e = cudaStreamWaitEvent(s, lane->copied[slot], 0);
    if (e != cudaSuccess) return cuda_fail(e, "streamed accumulate: copy");
    const char* Tg = static_cast<const char*>(T) + size_t(l0) * block_bytes;
    rc = run_batch_step(dst, dtype, nb, N, d, tsq + l0, eta, zero_first, xsq_total + l0, alpha + l0,
                        partials + size_t(l0) * size_t(sumsq_num_partials()), s);
    if (rc != LOCA_OK) return rc;
    rc = run_gram_cross(dst, Tg, dtype, nb, N, d, alpha + l0, zero_first, gram + size_t(l0) * dd,
                        cross + size_t(l0) * dd, flags, s);
    if (rc != LOCA_OK) return rc;
    e = cudaEventRecord(lane->consumed[slot], s);
    if (e != cudaSuccess) return cuda_fail(e, "streamed accumulate: event");
  }
  return LOCA_OK;
}

int loca_alignment_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (Np < 0 || m < 1 || d < 1 || L < 1 || r < 1)
    return fail(LOCA_ERR_SHAPE, "need Np >= 0, m, d, L, r >= 1");
  *bytes = align_workspace_bytes(Np, m, d, L, r);
  return LOCA_OK;
}

int loca_alignment(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d, int32_t L,
                   const float* P, const float* Q, int32_t r, double* alpha, void* workspace,
                   size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (Np < 0 || d < 1 || L < 1 || L > 65535 || Np > (int64_t(1) << 31))
    return fail(LOCA_ERR_SHAPE, "need 0 <= Np < 2^31, d >= 1, 1 <= L <= 65535");
  if (m < 1 || m > align_max_m()) return fail(LOCA_ERR_SHAPE, "need 1 <= m <= %d, got m=%d", align_max_m(), m);
  if (r < 1 || r > align_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got r=%d", align_max_r(), r);
  if ((Np > 0 && (!E_probe || !G_probe)) || !P || !Q || !alpha)
    return fail(LOCA_ERR_INVALID_ARG, "E_probe, G_probe, P, Q and alpha are required");
  if ((E_probe && !aligned(E_probe, 4)) || (G_probe && !aligned(G_probe, 4)) || !aligned(P, 4) || !aligned(Q, 4) ||
      !aligned(alpha, 8))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be aligned to their element size");
  const int rc = check_ws(workspace, workspace_bytes, align_workspace_bytes(Np, m, d, L, r));
  if (rc != LOCA_OK) return rc;
  cudaError_t e = launch_alignment(E_probe, G_probe, Np, m, d, L, P, Q, r, alpha, workspace,
                                   static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_alignment launch");
  return LOCA_OK;
}

int loca_kspace_workspace_size(int32_t L, int64_t N, int64_t d, int32_t k, int32_t C, int32_t r, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (L < 1 || N < 0 || d < 1 || k < 1 || k > 32 || C < 1 || C > kspace_max_C() || r < 1 || r > kspace_max_r())
    return fail(LOCA_ERR_SHAPE, "need L >= 1, N >= 0, d >= 1, 1 <= k <= 32, 1 <= C <= %d, 1 <= r <= %d",
                kspace_max_C(), kspace_max_r());
  *bytes = kspace_ws(L, N, d, k, C, r).total;
  return LOCA_OK;
}

int loca_kspace_accumulate(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const float* A, int32_t k,
                           const float* E, int32_t C, const float* P, const float* Q, int32_t r, float eta,
                           int zero_first, float* G, float* SC, double* xsq_total, float* alpha,
                           void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (dtype != LOCA_BF16) return fail(LOCA_ERR_UNSUPPORTED_DTYPE, "the k-space path takes bf16 X (dtype LOCA_BF16)");
  if (L < 1 || L > 65535 || N < 0 || N > 2147483647LL || d < 1 || d > 65536)
    return fail(LOCA_ERR_SHAPE, "need 1 <= L <= 65535, 0 <= N < 2^31, 1 <= d <= 65536");
  if (d % 8 != 0) return fail(LOCA_ERR_SHAPE, "need d %% 8 == 0 (16-byte rows), got d=%lld", (long long)d);
  if (k < 1 || k > 32 || k > d) return fail(LOCA_ERR_SHAPE, "need 1 <= k <= min(d, 32), got k=%d", k);
  if (C < 1 || C > kspace_max_C()) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= %d, got C=%d", kspace_max_C(), C);
  if (r < 1 || r > kspace_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got r=%d", kspace_max_r(), r);
  if (!(eta >= 0.f)) return fail(LOCA_ERR_INVALID_ARG, "eta must be >= 0");
  if ((N > 0 && (!X || !E)) || !A || !P || !Q || !G || !SC || !xsq_total)
    return fail(LOCA_ERR_INVALID_ARG, "X, A, E, P, Q, G, SC and xsq_total are required");
  if ((X && !aligned(X, 16)) || !aligned(A, 4) || (E && !aligned(E, 4)) || !aligned(P, 4) || !aligned(Q, 4) ||
      !aligned(G, 4) || !aligned(SC, 4) || !aligned(xsq_total, 8) || (alpha && !aligned(alpha, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "X needs 16-byte, xsq_total 8-byte, the other arrays 4-byte alignment");
  const KspaceWs lay = kspace_ws(L, N, d, k, C, r);
  int rc = check_ws(workspace, workspace_bytes, lay.total);
  if (rc != LOCA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  if (N == 0) {
    if (zero_first) {
      cudaError_t e = cudaMemsetAsync(G, 0, sizeof(float) * size_t(L) * k * k, s);
      if (e == cudaSuccess) e = cudaMemsetAsync(SC, 0, sizeof(float) * size_t(L) * C * k, s);
      if (e == cudaSuccess) e = cudaMemsetAsync(xsq_total, 0, sizeof(double) * size_t(L), s);
      if (e != cudaSuccess) return cuda_fail(e, "k-space accumulate: zeroing");
    }
    if (alpha) {
      cudaError_t e = cudaMemsetAsync(alpha, 0, sizeof(float) * size_t(L), s);
      if (e != cudaSuccess) return cuda_fail(e, "k-space accumulate: zeroing");
    }
    return LOCA_OK;
  }
  int32_t* status = device_status_word();
  if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  cudaError_t e = launch_kspace_accumulate(X, L, N, d, A, k, E, C, P, Q, r, eta, zero_first, G, SC, xsq_total,
                                           alpha, workspace, status, s);
  if (e != cudaSuccess) return cuda_fail(e, "k-space accumulate launch");
  return LOCA_OK;
}

int loca_kspace_solve(const float* G, const float* SC, const double* xsq_total, const float* P, const float* Q,
                      const float* B_prev, const float* lambda_rel, int32_t nl, int32_t L, int64_t d, int32_t k,
                      int32_t C, int32_t r, float* B, int32_t* info, float* C_out, void* stream) {
  g_msg[0] = 0;
  if (L < 1 || L > 65535 || d < 1) return fail(LOCA_ERR_SHAPE, "need 1 <= L <= 65535, d >= 1");
  if (k < 1 || k > 32 || k > d) return fail(LOCA_ERR_SHAPE, "need 1 <= k <= min(d, 32), got k=%d", k);
  if (C < 1 || C > kspace_max_C()) return fail(LOCA_ERR_SHAPE, "need 1 <= C <= %d, got C=%d", kspace_max_C(), C);
  if (r < 1 || r > kspace_max_r()) return fail(LOCA_ERR_SHAPE, "need 1 <= r <= %d, got r=%d", kspace_max_r(), r);
  if (nl < 1 || nl > 16) return fail(LOCA_ERR_SHAPE, "need 1 <= nl <= 16, got nl=%d", nl);
  if (!G || !SC || !P || !Q || !lambda_rel || !B || !info)
    return fail(LOCA_ERR_INVALID_ARG, "G, SC, P, Q, lambda_rel, B and info are required");
  for (int j = 0; j < nl; ++j)
    if (!(lambda_rel[j] > 0.f)) return fail(LOCA_ERR_INVALID_ARG, "lambda_rel[%d] must be > 0", j);
  if (!aligned(G, 4) || !aligned(SC, 4) || !aligned(P, 4) || !aligned(Q, 4) || !aligned(B, 4) || !aligned(info, 4) ||
      (B_prev && !aligned(B_prev, 4)) || (xsq_total && !aligned(xsq_total, 8)) || (C_out && !aligned(C_out, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be aligned to their element size");
  cudaError_t e = launch_kspace_solve(G, SC, xsq_total, P, Q, B_prev, lambda_rel, nl, L, d, k, C, r, B, info, C_out,
                                      static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "k-space solve launch");
  return LOCA_OK;
}

int loca_ridge_solve_workspace_size(int32_t L, int64_t d, int32_t k, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (L < 1 || d < 1 || k < 1) return fail(LOCA_ERR_SHAPE, "need L, d, k >= 1");
  *bytes = solve_ws(L, d, k).total;
  return LOCA_OK;
}

int loca_ridge_solve(const float* gram, const float* cross, const float* cross_scale, const double* xsq_total,
                     const float* A, const float* B_prev, const float* lambda_rel, int32_t nl, int32_t L,
                     int64_t d, int32_t k, float* B, int32_t* info, float* G_out, float* C_out,
                     void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (L < 1 || L > 65535 || d < 1) return fail(LOCA_ERR_SHAPE, "need 1 <= L <= 65535, d >= 1");
  if (k < 1 || k > 32 || k > d) return fail(LOCA_ERR_SHAPE, "need 1 <= k <= min(d, 32), got k=%d", k);
  if (nl < 1 || nl > 16) return fail(LOCA_ERR_SHAPE, "need 1 <= nl <= 16, got nl=%d", nl);
  if (!gram || !cross || !A || !lambda_rel || !B || !info)
    return fail(LOCA_ERR_INVALID_ARG, "gram, cross, A, lambda_rel, B and info are required");
  for (int j = 0; j < nl; ++j)
    if (!(lambda_rel[j] > 0.f)) return fail(LOCA_ERR_INVALID_ARG, "lambda_rel[%d] must be > 0", j);
  if (!aligned(gram, 4) || !aligned(cross, 4) || !aligned(A, 4) || !aligned(B, 4) ||
      !aligned(info, 4) || (B_prev && !aligned(B_prev, 4)) || (xsq_total && !aligned(xsq_total, 8)) ||
      (G_out && !aligned(G_out, 4)) || (C_out && !aligned(C_out, 4)) || (cross_scale && !aligned(cross_scale, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be aligned to their element size");
  const SolveWs lay = solve_ws(L, d, k);
  int rc = check_ws(workspace, workspace_bytes, lay.total);
  if (rc != LOCA_OK) return rc;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  float* GA = reinterpret_cast<float*>(ws_at(workspace, lay.ga));
  float* CA = reinterpret_cast<float*>(ws_at(workspace, lay.ca));
  cudaError_t e;
  int nsplit;
  if (project_tc_supported(gram, cross, A, d, k)) {
    int32_t* status = device_status_word();
    if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
    e = launch_project_tc(gram, cross, A, L, d, k, GA, CA, ws_at(workspace, lay.arec), status,
                          reinterpret_cast<int32_t*>(ws_at(workspace, lay.flag)), s);
    nsplit = 1;
  } else {
    e = launch_project_rows(gram, cross, A, L, d, k, GA, CA, s);
    nsplit = project_split();
  }
  if (e != cudaSuccess) return cuda_fail(e, "loca_ridge_solve: projection");
  e = launch_chol_solve(GA, CA, nsplit, A, B_prev, xsq_total, cross_scale, lambda_rel, nl, L, d, k, B, info, G_out,
                        C_out, reinterpret_cast<float*>(ws_at(workspace, lay.fac)), s);
  if (e != cudaSuccess) return cuda_fail(e, "loca_ridge_solve: solve");
  return LOCA_OK;
}

int loca_step_from_gram(const float* gram, int32_t L, int64_t d, const double* tsq, float eta, double* xsq_total,
                        float* alpha, void* stream) {
  g_msg[0] = 0;
  if (L < 1 || L > 65535 || d < 1) return fail(LOCA_ERR_SHAPE, "need 1 <= L <= 65535, d >= 1");
  if (!gram || !tsq || !xsq_total || !alpha)
    return fail(LOCA_ERR_INVALID_ARG, "gram, tsq, xsq_total and alpha are required");
  if (!aligned(gram, 4) || !aligned(tsq, 8) || !aligned(xsq_total, 8) || !aligned(alpha, 4))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be aligned to their element size");
  cudaError_t e = launch_step_from_gram(gram, L, d, tsq, eta, xsq_total, alpha, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_step_from_gram launch");
  return LOCA_OK;
}

int loca_calib_fit_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r, size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  if (Np < 1 || m < 1 || m > 64 || d < 1 || L < 1 || r < 1 || r > m)
    return fail(LOCA_ERR_SHAPE, "need Np >= 1, 1 <= r <= m <= 64, d >= 1, L >= 1");
  *bytes = calib_workspace_bytes(Np, m, d, L, r);
  return LOCA_OK;
}

int loca_calib_fit(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d,
                   int32_t L, float beta, int32_t r, float* P, float* Q, float* sigma,
                   void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  if (Np < 1 || m < 1 || m > 64 || d < 1 || L < 1 || L > 65535 || r < 1 || r > m)
    return fail(LOCA_ERR_SHAPE, "need Np >= 1, 1 <= r <= m <= 64, d >= 1, 1 <= L <= 65535");
  if (!(beta > 0.f)) return fail(LOCA_ERR_INVALID_ARG, "beta must be > 0");
  if (!E_probe || !G_probe || !P || !Q) return fail(LOCA_ERR_INVALID_ARG, "E_probe, G_probe, P and Q are required");
  if (!aligned(E_probe, 4) || !aligned(G_probe, 4) || !aligned(P, 4) || !aligned(Q, 4) ||
      (sigma && !aligned(sigma, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be 4-byte aligned");
  int rc = check_ws(workspace, workspace_bytes, calib_workspace_bytes(Np, m, d, L, r));
  if (rc != LOCA_OK) return rc;
  int32_t* status = device_status_word();
  if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  cudaError_t e = launch_calib_fit(E_probe, G_probe, Np, m, d, L, beta, r, P, Q, sigma, workspace,
                                   status, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_calib_fit launch");
  return LOCA_OK;
}

static int check_rsvd_shape(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r, int32_t ell) {
  const int64_t wmax = calib_rsvd_max_width();
  if (Np < 1 || Np > 65535LL * 64 || L < 1 || L > 65535 || r < 1 || ell < r || ell > calib_rsvd_max_ell() ||
      m < ell || d < ell || m > wmax || d > wmax)
    return fail(LOCA_ERR_SHAPE,
                "need 1 <= Np <= 4194240, 1 <= L <= 65535, 1 <= r <= ell <= %d, ell <= m <= %lld, ell <= d <= %lld",
                calib_rsvd_max_ell(), (long long)wmax, (long long)wmax);
  return LOCA_OK;
}

int loca_calib_fit_rsvd_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r, int32_t ell,
                                       size_t* bytes) {
  if (!bytes) return fail(LOCA_ERR_INVALID_ARG, "bytes is NULL");
  int rc = check_rsvd_shape(Np, m, d, L, r, ell);
  if (rc != LOCA_OK) return rc;
  *bytes = calib_rsvd_workspace_bytes(Np, m, d, L, ell, r);
  return LOCA_OK;
}

int loca_calib_fit_rsvd(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d, int32_t L,
                        float beta, int32_t r, int32_t ell, int32_t q, const float* Omega, float* P, float* Q,
                        float* sigma, void* workspace, size_t workspace_bytes, void* stream) {
  g_msg[0] = 0;
  int rc = check_rsvd_shape(Np, m, d, L, r, ell);
  if (rc != LOCA_OK) return rc;
  if (q < 0 || q > 16) return fail(LOCA_ERR_INVALID_ARG, "need 0 <= q <= 16 power iterations");
  if (!(beta > 0.f)) return fail(LOCA_ERR_INVALID_ARG, "beta must be > 0");
  if (!E_probe || !G_probe || !Omega || !P || !Q)
    return fail(LOCA_ERR_INVALID_ARG, "E_probe, G_probe, Omega, P and Q are required");
  if (!aligned(E_probe, 4) || !aligned(G_probe, 4) || !aligned(Omega, 4) || !aligned(P, 4) || !aligned(Q, 4) ||
      (sigma && !aligned(sigma, 4)))
    return fail(LOCA_ERR_ALIGNMENT, "pointers must be 4-byte aligned");
  rc = check_ws(workspace, workspace_bytes, calib_rsvd_workspace_bytes(Np, m, d, L, ell, r));
  if (rc != LOCA_OK) return rc;
  int32_t* status = device_status_word();
  if (!status) return fail(LOCA_ERR_CUDA, "cannot resolve the device status word");
  cudaError_t e = launch_calib_rsvd(E_probe, G_probe, Np, m, d, L, beta, r, ell, q, Omega, P, Q, sigma, workspace,
                                    status, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loca_calib_fit_rsvd launch");
  return LOCA_OK;
}

}  // extern "C"
