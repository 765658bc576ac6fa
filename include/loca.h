/*
 * loca.h — C ABI of the LoCA forward-only adaptation hot path on one GB300 (sm_103a).
 *
 * LoCA (Local Credit Assignment, arXiv 2608.03020) tunes the low-rank adapters
 * H_l = Hbar_l + B_l A_l H_{l-1} of a frozen transformer (Eq. 1) without further
 * backpropagation after one calibration.  One Stage-II outer iteration (S13) is, after
 * the forward pass:
 *
 *   loca_error        top-layer error at the frozen head             (Eq. 4, Lemma S3)
 *   loca_targets      tokenwise feedback predictions T_l = E P_l Q_l  (S3, S11)
 *   loca_accumulate   streamed Gram / cross statistics with the
 *                     scale-normalised step                          (Eqs. 6, 9, 10; S7, S8)
 *   loca_ridge_solve  projected statistics and positive-definite
 *                     solves B* = C (G + lambda I)^-1 for all blocks
 *                     and all ridge candidates                       (Eq. 8, Theorem S6, S7)
 *
 * and, once before Stage II, loca_calib_fit fits each block's rank-r feedback map from
 * probe-backward pairs (Eq. 5, S5).
 *
 * Notation: the paper's adapter rank (r) is k here and its feedback rank (k) is r here.
 * The head W_u restricted to the C label columns is folded into P_l, so the error E has
 * C columns and the paper's F_l e becomes the row  e^T P_l Q_l  (F_l^T = P_l Q_l).
 *
 * Conventions for every entry point:
 *  - All array arguments are DEVICE pointers owned by the caller, contiguous row-major,
 *    unless the argument's comment says "host".  The library allocates no memory; entry
 *    points that need scratch take a caller-provided device workspace whose size the
 *    matching *_workspace_size function returns (workspace may be NULL when that size
 *    is 0).  The workspace must not be shared by calls that may overlap on the GPU.
 *  - Work is enqueued asynchronously on `stream` (a cudaStream_t; NULL = the legacy
 *    default stream).  The return value reports host-side validation and launch errors
 *    only; conditions detected on the device (a bounded wait that gave up, see
 *    loca_device_status; a system that is not positive definite, see `info`) are written
 *    to device memory.
 *  - No exception crosses the ABI and nothing is printed.  loca_last_error_string()
 *    describes the last non-OK status of the calling thread.
 *  - Pointers to 16-bit or 32-bit data must be aligned to their element size; the bf16
 *    statistics path additionally needs 16-byte aligned X and T and d % 8 == 0 (its rows
 *    are fed to the tensor cores by TMA, which reads 16-byte rows).
 */
#ifndef LOCA_H_
#define LOCA_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
typedef enum loca_status {
  LOCA_OK = 0,
  LOCA_ERR_INVALID_ARG = 1,        /* null pointer where one is required, bad flag or value */
  LOCA_ERR_SHAPE = 2,              /* a size is out of range or inconsistent */
  LOCA_ERR_ALIGNMENT = 3,          /* a pointer or a row pitch is misaligned */
  LOCA_ERR_UNSUPPORTED_DTYPE = 4,  /* dtype code not accepted by this entry point */
  LOCA_ERR_CUDA = 5,               /* a CUDA runtime call or launch failed */
  LOCA_ERR_TIMEOUT = 6,            /* a device wait gave up (reported by loca_device_status) */
  LOCA_ERR_WORKSPACE = 7,          /* workspace missing or smaller than required */
  LOCA_ERR_UNSUPPORTED = 8,        /* valid request outside what this library supports */
  LOCA_ERR_NUMERIC = 9,            /* device: a system that should be positive definite was not
                                      in floating point (reported by loca_device_status) */
  LOCA_ERR_BOUNDS = 10             /* device, debug build only: an index left its buffer; the
                                      access was skipped (reported by loca_device_status) */
} loca_status;

/* Element type codes. */
enum { LOCA_F32 = 0, LOCA_BF16 = 1 };

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int loca_version(void);

/*
 * loca_set_wait_limit — test hook for the failure path (the paper has no counterpart).  Every
 * wait of the tensor-core kernels on an mbarrier (a copy landing, an MMA completing) is bounded;
 * when one runs out the kernel records LOCA_ERR_TIMEOUT in the device status word, makes the
 * other waits of its launch give up, lets the copies and MMAs already in flight land, frees its
 * tensor memory and returns, so the context stays usable.  This sets, for the whole process,
 * how long such a wait may take in the tensor-core kernels (loca_targets, loca_kspace_accumulate,
 * the CTA-pair Gram / cross kernel of loca_gram_cross, loca_accumulate and their variants, and the
 * projection of loca_ridge_solve)
 * before it gives up: ns = 0 restores the default of 4 s; a tiny value makes a call time out on
 * purpose, to test that path.
 */
int loca_set_wait_limit(uint64_t ns);

/* Message for the last non-OK status returned to the calling thread ("" if none). */
const char* loca_last_error_string(void);

/*
 * loca_device_status — read and clear the library's device status word on the current
 * device.  Kernels whose waits are bounded (the tensor-core statistics kernel) write
 * LOCA_ERR_TIMEOUT there when a wait gives up instead of hanging; their outputs are
 * then undefined.  Synchronises `stream`.  *host_status receives LOCA_OK or the code.
 */
int loca_device_status(int32_t* host_status /* host */, void* stream);

/*
 * Debug build (libloca_debug.so, compiled with -DLOCA_DEBUG; same entry points).  Every kernel
 * checks the index of each global access it computes, and the coordinates of its TMA stores,
 * against the extent of the buffer that the sizes of the call give.  A failed check skips the
 * access and records LOCA_ERR_BOUNDS with the source line; nothing traps.  loca_device_status
 * then returns LOCA_ERR_BOUNDS (after any code of the status word above) and names the source
 * file and line in loca_last_error_string().  The release library compiles the checks away.
 * loca_debug_build returns 1 in the debug build and 0 in the release build.
 */
int loca_debug_build(void);

/*
 * loca_error — top-layer error at the frozen head (Eq. 4; Lemma "Top-layer error", S3).
 *
 *   lse_n   = log sum_{j in S} exp(z[n, j])       S = full row (normaliser 0, the paper's
 *                                                 softmax over the vocabulary) or the
 *                                                 label columns (normaliser 1)
 *   E[n, c] = w_n (exp(z[n, label_cols[c]] - lse_n) - [y_n == c])
 *   ce[n]   = w_n (lse_n - z[n, label_cols[y_n]])
 *
 * logits      N x V, row pitch ldz elements (ldz >= V), LOCA_F32 or LOCA_BF16
 * label_cols  C int32 column indices in [0, V), C in [1, 1024]
 * y           N int32 labels in [0, C), or -1 for a masked position (weight 0, E row = 0)
 * w           N float loss weights w_n >= 0, or NULL for all ones
 * E           N x C float output
 * ce          N float output, or NULL
 * Arithmetic in fp32; one warp per row, single pass (running max and rescaled sum).
 */
int loca_error(const void* logits, int logit_dtype, int64_t N, int64_t V, int64_t ldz,
               const int32_t* label_cols, int32_t C, const int32_t* y, const float* w,
               int normaliser, float* E, float* ce, void* stream);

/*
 * loca_targets — tokenwise feedback predictions of every block (S3: Q_l := F_l E;
 * applied through the low-rank factors as in S11):  T_l = (E P_l) Q_l.
 *
 * E    N x C float (from loca_error)
 * P    L x C x r float, Q  L x r x d float (feedback factors, e.g. from loca_calib_fit)
 * T    L x N x d output, t_dtype LOCA_BF16 (the tensor-core feed) or LOCA_F32; 16-byte aligned
 * tsq  L double output ||T_l||_F^2 of the fp32 values before rounding, or NULL
 * Arithmetic: u = E[n] P_l in fp32; U Q_l on the tensor cores (tcgen05, kind::tf32) as
 * hi*hi + hi*lo + lo*hi of tf32 splits with fp32 accumulation (fp32-accurate); one rounding
 * to the output type.  r in [1, 32], C in [1, 64].  A workspace is always required (it also
 * holds a launch-local wait flag).  Deterministic: partial sums are reduced in a fixed order.
 */
int loca_targets_workspace_size(int64_t N, int32_t L, int64_t d, size_t* bytes /* host */);
int loca_targets(const float* E, int64_t N, int32_t C, const float* P, const float* Q,
                 int32_t L, int32_t r, int64_t d, void* T, int t_dtype, double* tsq,
                 void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_accumulate — add one mini-batch of N tokens to the sufficient statistics of every
 * block (Eqs. 6 and 9; additivity over mini-batches, S7; one step per block and
 * mini-batch, Eq. 10 and S8):
 *
 *   xsq_b[l]  = ||X_l||_F^2                              (this batch)
 *   alpha_l   = -eta sqrt(xsq_b[l] / tsq[l]), 0 if tsq[l] == 0
 *               (= -eta_bar: eta RMS(X_l) / RMS(T_l), both N x d)
 *   gram_l   += X_l^T X_l                                (d x d, symmetric, both halves written)
 *   cross_l  += alpha_l T_l^T X_l                        (d x d; row = output channel i,
 *                                                        column = input channel j)
 *   xsq_total[l] += xsq_b[l]
 *
 * With zero_first != 0 the three outputs are overwritten instead of accumulated.
 * X, T  L x N x d, both of `dtype`:
 *   LOCA_BF16  tcgen05 tensor-core GEMM, bf16 operands, fp32 accumulation in tensor
 *              memory; needs d % 8 == 0 and 16-byte aligned X and T
 *   LOCA_F32   exact-input path: fp32 operands, fp64 accumulation (slow; small shapes)
 * tsq   L double (from loca_targets, over the same tokens)
 * gram, cross  L x d x d float;  xsq_total  L double.
 * Deterministic: every output element is produced by one thread in a fixed order.
 */
int loca_accumulate_workspace_size(int32_t L, int64_t N, int64_t d, int dtype,
                                   size_t* bytes /* host */);
int loca_accumulate(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                    const double* tsq, float eta, int zero_first, float* gram, float* cross,
                    double* xsq_total, void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_accumulate_streamed — loca_accumulate with X read from host memory (Eqs. 6, 9, 10; S7,
 * S8: the same statistics, the same results).  For activations kept in host memory (a
 * calibration set larger than device memory, or a producer on the CPU side): X_host is copied
 * to the device group by group of `group` blocks and the statistics of group g run while group
 * g + 1 is being copied, so the copy time and the kernel time overlap instead of adding up.
 *
 * X_host   L x N x d host array of `dtype` (page-locked memory gives the full copy rate;
 *          pageable memory works, but the driver stages each copy and the call then waits for
 *          it on the host).
 * staging  device array of at least 2 x group x N x d elements of `dtype`, 16-byte aligned: two
 *          copy slots used alternately; on return it holds the last one or two groups.
 * group    blocks per copy (1 <= group; values above L are clamped to L).
 * T, tsq, eta, zero_first, gram, cross, xsq_total, dtype, workspace: as loca_accumulate
 *          (workspace size: loca_accumulate_workspace_size).
 *
 * Ordering: the kernels run on `stream`, each after the copy of its group.  The copies run
 * on a copy stream that the library creates on the first call on each device (with four
 * events; no device memory is allocated).  A copy into a slot waits for the kernels that last
 * read that slot (in this or an earlier call), but not for any other work on `stream`: the
 * caller must not let other queued work read or write `staging`.  X_host must stay valid and
 * unchanged until the copies have run (synchronise `stream` before reusing it).
 */
int loca_accumulate_streamed(const void* X_host, void* staging, const void* T, int dtype, int32_t L,
                             int64_t N, int64_t d, int32_t group, const double* tsq, float eta,
                             int zero_first, float* gram, float* cross, double* xsq_total,
                             void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_alignment — in-probe alignment diagnostic of the feedback map (supplement, one-shot
 * calibration; S5): for every block,
 *   alpha[l] = <G_l, T_l>_F / (||G_l||_F ||T_l||_F),   T_l = E_probe P_l Q_l,
 * the cosine between the stacked feedback predictions and the stacked exact hidden-state
 * gradients at the probe positions (0 when either is zero).  Random feedback gives ~0; the
 * paper reports 0.3-0.5 after calibration.
 *   E_probe  Np x m float (m <= 16384);  G_probe  L x Np x d float;  P  L x m x r,
 *   Q  L x r x d float (r <= 32);  alpha  L double (output).
 *   Workspace: loca_alignment_workspace_size (partial sums; for m > 64, the paper's d-wide
 *   error space, also U_l = E_probe P_l, L x Np x r float, formed first).
 *   T is formed in registers and never written; sums in fp32 per thread over 1024 tokens,
 *   fp64 across, in a fixed order (deterministic).
 */
int loca_alignment_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r,
                                  size_t* bytes /* host */);
int loca_alignment(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d,
                   int32_t L, const float* P, const float* Q, int32_t r, double* alpha,
                   void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_kspace_accumulate / loca_kspace_solve — the paper's own statistics in adapter space
 * (Eqs. 6, 8, 9; S7, S8) instead of the d x d Gram and cross product: the same solved system
 * (Theorem S6), O(L (k^2 + C k)) state, and one HBM read of X per block and mini-batch.
 *
 * loca_kspace_accumulate, for every block l, with p_n = A_l^T x_n (Eq. 9's features) and the
 * targets q_n = (e_n P_l) Q_l applied through the factors (S3, S11; T is never formed):
 *   xsq_b[l]  = ||X_l||_F^2;   tsq_b[l] = sum_n ||q_n||^2 = sum_n u_n^T (Q_l Q_l^T) u_n, u_n = e_n P_l
 *   alpha[l]  = -eta sqrt(xsq_b[l] / tsq_b[l])  (0 if tsq_b[l] == 0; = -eta_bar, Eq. 10, S8)
 *   G_l      (+)= sum_n p_n p_n^T                       (k x k)
 *   SC_l     (+)= alpha[l] sum_n e_n p_n^T              (C x k)
 *   xsq_total[l] (+)= xsq_b[l]
 * so that C_l = B_prev,l G_l + Q_l^T (P_l^T SC_l) = sum_n rho_n p_n^T with
 * rho_n = B_prev p_n - eta_bar q_n (Eq. 6).  zero_first != 0 overwrites instead of adding.
 *   X  L x N x d bf16 (LOCA_BF16 only), 16-byte aligned, d % 8 == 0;  A  L x d x k float (k <= 32);
 *   E  N x C float (C <= 16);  P  L x C x r float, Q  L x r x d float (r <= 32);
 *   G  L x k x k float;  SC  L x C x k float;  xsq_total  L double;  alpha  L float or NULL.
 *   Workspace: loca_kspace_workspace_size (the split A_l, Q_l Q_l^T, per-CTA partial sums and
 *   E^T E partials; 2 KB per 1024 tokens beyond a fixed part).
 *   Arithmetic: X A_l on the tensor cores with A_l split into two bf16 parts (A_l to 2^-16) and
 *   fp32 accumulation; the token sums in fp32 over 128 tokens, fp64 across; fixed-order
 *   reductions (deterministic).
 *
 * loca_kspace_solve (Eq. 8; Theorem S6; S7): for every candidate j and block l,
 *   lambda_{j,l} = lambda_rel[j] * xsq_total[l] / d  (absolute lambda_rel if xsq_total == NULL),
 *   B[j, l] = C_l (G_l + lambda I)^-1 by Cholesky (no inverse), C_l as above.
 *   lambda_rel: nl host floats (nl <= 16, each > 0); B: nl x L x d x k float; info: nl x L int32
 *   (0, or the order of the first non-positive leading minor; then B[j, l] is zero);
 *   B_prev: L x d x k or NULL (= 0); C_out: L x d x k or NULL.
 */
int loca_kspace_workspace_size(int32_t L, int64_t N, int64_t d, int32_t k, int32_t C, int32_t r,
                               size_t* bytes /* host */);
int loca_kspace_accumulate(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const float* A,
                           int32_t k, const float* E, int32_t C, const float* P, const float* Q,
                           int32_t r, float eta, int zero_first, float* G, float* SC,
                           double* xsq_total, float* alpha, void* workspace, size_t workspace_bytes,
                           void* stream);
int loca_kspace_solve(const float* G, const float* SC, const double* xsq_total, const float* P,
                      const float* Q, const float* B_prev, const float* lambda_rel /* host */,
                      int32_t nl, int32_t L, int64_t d, int32_t k, int32_t C, int32_t r, float* B,
                      int32_t* info, float* C_out, void* stream);

/*
 * loca_host_alloc / loca_host_free — host memory for inputs streamed to the GPU (for example
 * X_host of loca_accumulate_streamed).  The paper has no counterpart: this concerns only the
 * speed of host-to-device copies.  Page-locked memory with 4 KiB pages copies at a rate that
 * varies widely once buffers reach tens of GB; this memory is backed by 2 MiB pages (anonymous
 * mapping, transparent huge pages advised, touched once in parallel) and registered with CUDA,
 * and copies at the full link rate.  Contents start at zero.  The size is rounded up to a
 * multiple of 2 MiB.  Free with loca_host_free (it unregisters and unmaps); a pointer not
 * returned by loca_host_alloc is rejected with LOCA_ERR_INVALID_ARG.  Needs a CUDA device.
 */
int loca_host_alloc(size_t bytes, void** ptr /* host, out */);
int loca_host_free(void* ptr);

/*
 * loca_batch_step and loca_gram_cross — the two halves of loca_accumulate, for callers that
 * schedule them separately (for example to time the tensor-core kernel on its own).
 *
 * loca_batch_step (Eq. 10; S8): xsq_b[l] = ||X_l||_F^2, alpha[l] = -eta sqrt(xsq_b[l] / tsq[l])
 *   (0 if tsq[l] == 0), xsq_total[l] = (zero_first ? 0 : xsq_total[l]) + xsq_b[l].
 *   alpha: L float device output.  Workspace: loca_batch_step_workspace_size.
 * loca_gram_cross (Eq. 9; S7): gram_l (+)= X_l^T X_l, cross_l (+)= alpha[l] T_l^T X_l with the
 *   alpha of loca_batch_step.  Workspace: loca_gram_cross_workspace_size (256 bytes; holds
 *   launch-local flags).  Arguments, layouts, dtypes and determinism as loca_accumulate.
 */
int loca_batch_step_workspace_size(int32_t L, size_t* bytes /* host */);
int loca_batch_step(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const double* tsq,
                    float eta, int zero_first, double* xsq_total, float* alpha, void* workspace,
                    size_t workspace_bytes, void* stream);
int loca_gram_cross_workspace_size(size_t* bytes /* host */);
int loca_gram_cross(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                    const float* alpha, int zero_first, float* gram, float* cross, void* workspace,
                    size_t workspace_bytes, void* stream);

/*
 * Fused targets: the Gram / cross statistics with each block's targets generated inside the
 * tensor-core kernel instead of read from memory (S3: Q_l := F_l E; S11: F e applied through
 * the factors).  Together with loca_targets_sq they replace loca_targets + loca_gram_cross; T is
 * never written, so the statistics read only X from HBM.
 *
 * loca_targets_sq (S3, S11; the ||Q_l||^2 of the step in Eq. 10):
 *   tsq[l] = ||E P_l Q_l||_F^2 = < P_l (Q_l Q_l^T) P_l^T , E^T E >, without forming T.
 *   E N x C, P L x C x r, Q L x r x d (fp32, row-major, device); tsq L doubles (device, out).
 *   1 <= C <= 64, 1 <= r <= 32.  fp32 products summed in fp64; deterministic.
 *   Workspace: loca_targets_sq_workspace_size(N, C) bytes (partial sums of E^T E).
 * loca_gram_cross_fused (Eq. 9; S7): gram_l (+)= X_l^T X_l, cross_l (+)= alpha[l] T_l^T X_l with
 *   T_l = (E P_l) Q_l formed tile by tile on the tensor cores (bf16 hi / lo parts of U = E P_l and
 *   of Q_l, three products, ~2^-17 per element) and rounded once to bf16 before it meets X, as
 *   loca_gram_cross does with a T from loca_targets.  X: L x N x d bf16 only (dtype LOCA_BF16),
 *   E, P, Q as loca_targets_sq, 1 <= r <= 32, C <= 64.  Workspace:
 *   loca_gram_cross_fused_workspace_size(L, N, r) bytes (launch-local flags and U_l = E P_l as
 *   bf16 hi / lo parts, 4 L N rp bytes with rp = 16 for r <= 16, else 32).  Other arguments,
 *   layouts and determinism as loca_gram_cross.
 *   Cost: the cross tiles take one accumulator each (the T generation needs the other TMEM
 *   half), so this kernel does more passes over X than loca_gram_cross; it saves the write of
 *   T and its reads.
 */
int loca_targets_sq_workspace_size(int64_t N, int32_t C, size_t* bytes /* host */);
int loca_targets_sq(const float* E, int64_t N, int32_t C, const float* P, const float* Q, int32_t L, int32_t r,
                    int64_t d, double* tsq, void* workspace, size_t workspace_bytes, void* stream);
int loca_gram_cross_fused_workspace_size(int32_t L, int64_t N, int32_t r, size_t* bytes /* host */);
int loca_gram_cross_fused(const void* X, int dtype, int32_t L, int64_t N, int64_t d, const float* E, int32_t C,
                          const float* P, const float* Q, int32_t r, const float* alpha, int zero_first,
                          float* gram, float* cross, void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_accumulate_noalloc — loca_accumulate for callers that cannot provide device scratch
 * memory.  The paper has no counterpart: it concerns only how this library obtains scratch.
 *
 * Some callers cannot allocate device memory when they call the library: a program whose
 * device memory is reserved up front by another owner (an inference server, a plugin host
 * that exposes no allocator), or a caller that must not call cudaMalloc on its hot loop
 * because the call can synchronise the device and take an unbounded time.  This entry point
 * allocates nothing: its scratch (partial sums of ||X_l||^2, the steps alpha_l and a wait
 * flag; 524,800 bytes) is a fixed array in the library's device memory that every GPU which
 * loads the library holds until the process exits.  Arguments, outputs and results are
 * those of loca_accumulate, without the workspace.
 *
 * Limits and use:
 *  - L <= 64 blocks; a larger L is rejected with LOCA_ERR_SHAPE (use loca_accumulate).
 *  - Every call looks up the array's device address in the current context
 *    (cudaGetSymbolAddress, with the caller's device current; the lookup allocates nothing and
 *    stays valid after a cudaDeviceReset).  The first lookup on a device may load the library's
 *    device code there: make the first call on each device before any stream capture.
 *  - Every call reuses the same array.  Calls whose work may overlap on the GPU (different
 *    streams, or threads without ordering between them) race on it: serialise them.
 *  - Calls no cudaMalloc, cudaFree or other allocating routine.
 */
int loca_accumulate_noalloc(const void* X, const void* T, int dtype, int32_t L, int64_t N, int64_t d,
                            const double* tsq, float eta, int zero_first, float* gram, float* cross,
                            double* xsq_total, void* stream);

/*
 * loca_step_from_gram — the step of Eq. 10 for a pass with one mini-batch, without reading X:
 * that batch's Gram (loca_gram_cross with zero_first = 1) holds X_l^T X_l, whose trace is
 * ||X_l||_F^2, so
 *
 *   xsq_total[l] = tr(gram_l),   alpha[l] = -eta sqrt(xsq_total[l] / tsq[l])   (0 if tsq[l] == 0)
 *
 * (RMS ratio of Eq. 10; N d cancels).  With the cross product accumulated at alpha = 1, pass
 * alpha to loca_ridge_solve as cross_scale: the same C_l as loca_batch_step + loca_gram_cross.
 * gram  L x d x d float (device); tsq  L double; xsq_total  L double (output); alpha  L float
 * (output).  The trace is summed in fp64 in a fixed order.  Only valid when gram holds exactly
 * one mini-batch; for several, use loca_batch_step before each loca_gram_cross.
 */
int loca_step_from_gram(const float* gram, int32_t L, int64_t d, const double* tsq, float eta,
                        double* xsq_total, float* alpha, void* stream);

/*
 * loca_ridge_solve — closed-form block minimisers for every block l and every ridge
 * candidate j (Eq. 8; Theorem S6; positive-definite solve without an inverse, S7):
 *
 *   G_l   = A_l^T gram_l A_l                              (k x k, Eq. 9 with p = A_l^T x)
 *   C_l   = B_prev,l G_l + s_l cross_l A_l                (d x k; = sum_n rho_n p_n^T with
 *                                                         rho = B^(t) p - eta_bar q, Eq. 6)
 *   s_l   = cross_scale[l], or 1 when cross_scale is NULL (a pass with one mini-batch may
 *           accumulate cross with alpha = 1 and apply alpha_l here; see loca_step_from_gram)
 *   lam   = lambda_rel[j] * xsq_total[l] / d              (xsq_total != NULL; = tr(gram_l)/d)
 *         = lambda_rel[j]                                 (xsq_total == NULL: absolute)
 *   B[j, l] = C_l (G_l + lam I)^-1   via Cholesky (fp64) and two triangular substitutions
 *
 * gram, cross   L x d x d float;  cross_scale  L float (device) or NULL
 * A             L x d x k float;  B_prev  L x d x k float or NULL (0)
 * lambda_rel    HOST array of nl > 0 positive floats, nl <= 16
 * B             nl x L x d x k float output;  info  nl x L int32 output: 0, or p > 0 when
 *               the p-th pivot of G_l + lam I is not positive (B[j, l] is then zero)
 * G_out         L x k x k float output or NULL;  C_out  L x d x k float output or NULL
 * 1 <= k <= min(d, 32); 1 <= nl <= 16.
 * The products gram_l A_l and cross_l A_l run on the tensor cores when d and k are multiples of
 * 4 and gram, cross and A are 16-byte aligned, else on the CUDA cores in fp32.  On the tensor
 * cores each operand is split into two fp16 parts after scaling by a power of two per
 * 32-channel row slice (gram, cross) or column slice (A), which carries every value to within
 * 2^-22 of itself; the part products are exact in fp32 and summed in fp32, as accurate as an
 * fp32 FMA evaluation.  The tensor-core
 * path's waits are bounded (loca_set_wait_limit); one that gives up writes LOCA_ERR_TIMEOUT to
 * the device status word and leaves B undefined.
 */
int loca_ridge_solve_workspace_size(int32_t L, int64_t d, int32_t k, size_t* bytes /* host */);
int loca_ridge_solve(const float* gram, const float* cross, const float* cross_scale,
                     const double* xsq_total, const float* A, const float* B_prev,
                     const float* lambda_rel /* host */,
                     int32_t nl, int32_t L, int64_t d, int32_t k, float* B, int32_t* info,
                     float* G_out, float* C_out, void* workspace, size_t workspace_bytes,
                     void* stream);

/*
 * loca_calib_fit — one-shot reduced-rank fit of every block's feedback map from
 * probe-backward pairs (Eq. 5; Theorem "Feedback ridge solution" and Lemma
 * "Rank-truncation error", S5).  Token-major:
 *
 *   F_hat_l^T = (E_probe^T E_probe + beta I_m)^-1 E_probe^T G_probe_l      (m x d)
 *   F_hat_l^T = U S V^T  (thin SVD),  P_l = U_r S_r (m x r),  Q_l = V_r^T (r x d)
 *
 * so that loca_targets with (P_l, Q_l) applies the rank-r map F_l = (P_l Q_l)^T.  Signs:
 * the entry of largest magnitude in each row of Q_l is positive.  Singular values that
 * are zero (r > rank) give zero rows of Q_l and zero columns of P_l.
 *
 * E_probe  Np x m float; G_probe  L x Np x d float; beta > 0; 1 <= r <= m <= 64
 * P        L x m x r float; Q  L x r x d float; sigma  L x r float or NULL
 * Arithmetic: E^T E and E^T G_l from fp32 products summed in fp32 over 32-token chunks and in
 * fp64 across chunks; Cholesky solve (fp64) for F_hat^T; cyclic Jacobi eigen-decomposition
 * (fp64) of the m x m matrix F_hat^T F_hat, whose eigenvectors are U and whose eigenvalues are
 * S^2; Q_l = S_r^-1 U_r^T F_hat^T.  Singular values below 1e-12 sigma_1 count as zero.  If
 * E^T E + beta I is not positive definite in floating point (beta below the rounding level
 * of E^T E), LOCA_ERR_NUMERIC is written to the device status word and that block's P, Q and
 * sigma are zero.
 */
int loca_calib_fit_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r,
                                  size_t* bytes /* host */);
int loca_calib_fit(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d,
                   int32_t L, float beta, int32_t r, float* P, float* Q, float* sigma,
                   void* workspace, size_t workspace_bytes, void* stream);

/*
 * loca_calib_fit_rsvd — the rank-r feedback fit of loca_calib_fit for error spaces too wide
 * to form and decompose F_hat_l^T (m x d), e.g. the paper's e = W_u^T eps with m = d (Eq. 5;
 * Theorem "Feedback ridge solution" and Lemma "Rank-truncation error", S5).  The top-r SVD
 * of F_hat_l^T = (E^T E + beta I_m)^-1 E^T G_l comes from randomized subspace iteration
 * (Halko, Martinsson and Tropp, SIAM Review 53 (2011), Algorithm 4.4 with q power
 * iterations, then Algorithm 5.1), which applies F_hat^T and F_hat only to ell vectors at a
 * time through a Cholesky factor of E^T E + beta I (shared by all blocks; no inverse):
 *
 *   Y = F^T Omega, Q_Y = orth(Y); q times: Z = orth(F Q_Y), Q_Y = orth(F^T Z);
 *   B = Q_Y^T F^T = U_B S V^T;  P_l = Q_Y U_B,r S_r (m x r),  Q_l = V_r^T (r x d).
 *
 * It equals loca_calib_fit's result when ell >= rank(F_hat_l^T); otherwise its error
 * approaches the truncated SVD's as (sigma_{ell+1} / sigma_r)^(2q+1).  Same sign convention
 * and zero threshold as loca_calib_fit.
 *
 * E_probe  Np x m float; G_probe  L x Np x d float; beta > 0
 * Omega    d x ell float, device: the caller's Gaussian test matrix, used for every block
 * 1 <= r <= ell <= 64, ell <= m <= 16384, ell <= d <= 16384, 0 <= q <= 16, 1 <= L <= 65535,
 * 1 <= Np <= 4194240
 * P        L x m x r float; Q  L x r x d float; sigma  L x r float or NULL
 * Arithmetic: products with E and G_l from fp32 products summed in fp32 over 128-term runs
 * and in fp64 across runs; Cholesky factor, triangular solves, orthonormal bases (Gram-Schmidt
 * with re-orthogonalisation) and the Rayleigh-Ritz step in fp64.  Workspace (device, at least
 * loca_calib_fit_rsvd_workspace_size bytes, 256-byte aligned) holds E^T E (m x m fp64,
 * m rounded up to 64) and the ell-column blocks of every block; its contents are scratch.
 * If E^T E + beta I is not positive definite in floating point, LOCA_ERR_NUMERIC is written
 * to the device status word and P, Q and sigma are zero.
 */
int loca_calib_fit_rsvd_workspace_size(int64_t Np, int32_t m, int64_t d, int32_t L, int32_t r,
                                       int32_t ell, size_t* bytes /* host */);
int loca_calib_fit_rsvd(const float* E_probe, const float* G_probe, int64_t Np, int32_t m, int64_t d,
                        int32_t L, float beta, int32_t r, int32_t ell, int32_t q, const float* Omega,
                        float* P, float* Q, float* sigma, void* workspace, size_t workspace_bytes,
                        void* stream);

#ifdef __cplusplus
}
#endif

#endif /* LOCA_H_ */
