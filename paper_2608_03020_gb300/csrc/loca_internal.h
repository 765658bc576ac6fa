// Internal declarations shared by the library's translation units (host side).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/loca.h"
#include "debug_check.cuh"

namespace loca {

// Number of SMs of the current device (cached per device).
int sm_count();

// Device address of the library's status word on the current device (see
// loca_device_status); resolved once per device with that device current.
int32_t* device_status_word();

// cuTensorMapEncodeTiled from the driver (looked up once), or nullptr.
typedef CUresult (*TensorMapEncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                      const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                      const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                      CUtensorMapL2promotion, CUtensorMapFloatOOBfill);
TensorMapEncodeFn tensor_map_encoder();

// Record the message loca_last_error_string() returns for the calling thread; returns `code`.
int set_error_message(int code, const char* fmt, ...);

// Bytes needed to round `n` up to a 256-byte boundary.
inline size_t align256(size_t n) { return (n + 255) & ~size_t(255); }

// ---- head error (error.cu)
cudaError_t launch_head_error(const void* z, int dtype, int64_t N, int64_t V, int64_t ldz,
                              const int32_t* cols, int C, const int32_t* y, const float* w,
                              int normaliser, float* E, float* ce, cudaStream_t s);

// ---- feedback targets (targets.cu)
// Workspace: partial sums of ||T_l||^2 (L x targets_num_partials(N, d) doubles) and a
// launch-local wait flag; targets_workspace_bytes gives the total.
int64_t targets_num_partials(int64_t N, int64_t d);
size_t targets_workspace_bytes(int64_t N, int L, int64_t d);
int targets_max_C();
int targets_max_r();
cudaError_t launch_targets(const float* E, int64_t N, int C, const float* P, const float* Q,
                           int L, int r, int64_t d, void* T, int t_dtype, double* tsq,
                           void* workspace, int32_t* status, cudaStream_t s);

// ---- statistics (stats.cu, gram_tc.cu)
// Sum of squares of X (per block) and the step alpha_l; partials: L x sumsq_num_partials().
int sumsq_num_partials();
cudaError_t launch_sumsq_and_step(const void* X, int dtype, int L, int64_t N, int64_t d,
                                  const double* tsq, float eta, int zero_first, double* xsq_total,
                                  double* partials, float* alpha, cudaStream_t s);
// alpha_l and xsq_total[l] from tr(Gram_l) of a pass with one mini-batch (no read of X).
cudaError_t launch_step_from_gram(const float* gram, int L, int64_t d, const double* tsq, float eta,
                                  double* xsq_total, float* alpha, cudaStream_t s);
// fp32-input Gram / cross (fp64 accumulation).
cudaError_t launch_gram_cross_f32(const float* X, const float* T, int L, int64_t N, int64_t d,
                                  const float* alpha, int zero_first, float* gram, float* cross,
                                  cudaStream_t s);
// bf16-input Gram / cross on tcgen05 tensor cores.  abort_flag points to two int32 of launch-local
// device memory (abort flag, round counter), both reset by the launcher on stream s.
cudaError_t launch_gram_cross_tc(const void* X, const void* T, int L, int64_t N, int64_t d,
                                 const float* alpha, int zero_first, float* gram, float* cross,
                                 int32_t* status, int32_t* abort_flag, cudaStream_t s);

// Gram / cross with the targets generated in the kernel from E, P, Q (bf16 X only); r <= 32.
// Workspace: launch-local flags (256 bytes), then U_l = E P_l as bf16 hi / lo parts.
int gram_fused_max_r();
size_t gram_fused_workspace_bytes(int L, int64_t N, int r);
cudaError_t launch_gram_cross_fused_tc(const void* X, const float* E, int C, const float* P, const float* Q,
                                       int r, int L, int64_t N, int64_t d, const float* alpha, int zero_first,
                                       float* gram, float* cross, int32_t* status, void* workspace,
                                       cudaStream_t s);
// ||T_l||^2 in closed form (targets_sq.cu); workspace: tsq_workspace_bytes(N, C).
int tsq_max_C();
int tsq_max_r();
size_t tsq_workspace_bytes(int64_t N, int C);
cudaError_t launch_targets_sq(const float* E, int64_t N, int C, const float* P, const float* Q, int L, int r,
                              int64_t d, double* tsq, void* workspace, cudaStream_t s);

// Host-side checks and launches shared by the statistics entry points (loca_abi.cu): they set the
// message of loca_last_error_string() and return a loca_status.
int validate_stats_inputs(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                          bool need_T);
int validate_accumulate(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                        const double* tsq, float eta, const float* gram, const float* cross,
                        const double* xsq_total);
int run_batch_step(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const double* tsq,
                   float eta, int zero_first, double* xsq_total, float* alpha, double* partials,
                   cudaStream_t s);
int run_gram_cross(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                   const float* alpha, int zero_first, float* gram, float* cross, int32_t* abort_flag,
                   cudaStream_t s);

// Limit of the bounded device waits of the tensor-core kernels (targets, k-space statistics,
// Gram / cross): 4 s unless loca_set_wait_limit changed it.
unsigned long long wait_limit_ns();

// ---- alignment diagnostic (align.cu)
int align_max_m();
int align_max_r();
size_t align_workspace_bytes(int64_t Np, int m, int64_t d, int L, int r);
cudaError_t launch_alignment(const float* E, const float* G, int64_t Np, int m, int64_t d, int L, const float* P,
                             const float* Q, int r, double* alpha, void* workspace, cudaStream_t s);

// ---- k-space statistics and solve (kspace.cu)
struct KspaceWs {
  size_t W, M, part, ete, flags, total;
};
KspaceWs kspace_ws(int L, int64_t N, int64_t d, int k, int C, int r);
int kspace_max_C();
int kspace_max_r();
cudaError_t launch_kspace_accumulate(const void* X, int L, int64_t N, int64_t d, const float* A, int k,
                                     const float* E, int C, const float* P, const float* Q, int r, float eta,
                                     int zero_first, float* G, float* SC, double* xsq_total, float* alpha_out,
                                     void* workspace, int32_t* status, cudaStream_t s);
cudaError_t launch_kspace_solve(const float* G, const float* SC, const double* xsq_total, const float* P,
                                const float* Q, const float* B_prev, const float* lambda_rel, int nl, int L,
                                int64_t d, int k, int C, int r, float* B, int32_t* info, float* C_out,
                                cudaStream_t s);

// ---- ridge solve (solve.cu, project_tc.cu)
// k_project_rows writes GA / CA as project_split() partial products each (L x d x k fp32 apiece);
// the tensor-core projection writes one (nsplit = 1).  The solve sums the nsplit partials.
int project_split();
cudaError_t launch_project_rows(const float* gram, const float* cross, const float* A, int L,
                                int64_t d, int k, float* GA, float* CA, cudaStream_t s);
// Tensor-core projection (fp16 MMAs on a row- and column-scaled two-part split): d % 4 == 0,
// k % 4 == 0, 4 <= k <= 32, 16-byte aligned gram, cross and A.  arec: project_tc_workspace_bytes
// of 16-byte aligned device memory for A's split slabs; abort_flag: 4 bytes of launch-local
// device memory.
bool project_tc_supported(const float* gram, const float* cross, const float* A, int64_t d, int k);
size_t project_tc_workspace_bytes(int L, int64_t d, int k);
cudaError_t launch_project_tc(const float* gram, const float* cross, const float* A, int L, int64_t d, int k,
                              float* GA, float* CA, void* arec, int32_t* status, int32_t* abort_flag,
                              cudaStream_t s);
// fac: chol_workspace_bytes(L) of device memory for the per-candidate factors (nl <= 16).
size_t chol_workspace_bytes(int L);
cudaError_t launch_chol_solve(const float* GA, const float* CA, int nsplit, const float* A, const float* B_prev,
                              const double* xsq_total, const float* cross_scale, const float* lambda_rel,
                              int nl, int L, int64_t d, int k, float* B, int32_t* info, float* G_out,
                              float* C_out, float* fac, cudaStream_t s);

// ---- calibration (calib.cu)
size_t calib_workspace_bytes(int64_t Np, int m, int64_t d, int L, int r);
cudaError_t launch_calib_fit(const float* E_probe, const float* G_probe, int64_t Np, int m,
                             int64_t d, int L, float beta, int r, float* P, float* Q, float* sigma,
                             void* workspace, int32_t* status, cudaStream_t s);

// ---- calibration for wide error spaces, randomized subspace iteration (calib_rsvd.cu)
int calib_rsvd_max_ell();
int64_t calib_rsvd_max_width();
size_t calib_rsvd_workspace_bytes(int64_t Np, int64_t m, int64_t d, int L, int ell, int r);
cudaError_t launch_calib_rsvd(const float* E_probe, const float* G_probe, int64_t Np, int64_t m, int64_t d, int L,
                              float beta, int r, int ell, int q, const float* Omega, float* P, float* Q,
                              float* sigma, void* workspace, int32_t* status, cudaStream_t s);

}  // namespace loca
