"""Python binding of ``libloca.so`` (argument marshalling only).

Every function here has the name of the C entry point it calls (``include/loca.h``), checks
the tensors it is given (device, dtype, shape, contiguity), passes their device pointers and
the current torch stream, and raises :class:`LocaError` on a non-OK status.  All arithmetic
of the hot path runs in the library's CUDA kernels; PyTorch only provides device memory and
streams.  There is no CPU fallback: importing works without a GPU, calling needs one.
"""

from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libloca.so")
LIB_DEBUG_PATH = os.path.join(_PKG, "libloca_debug.so")  # built with -DLOCA_DEBUG (bounds checks)

LOCA_F32 = 0
LOCA_BF16 = 1

STATUS_NAMES = {
    0: "LOCA_OK", 1: "LOCA_ERR_INVALID_ARG", 2: "LOCA_ERR_SHAPE", 3: "LOCA_ERR_ALIGNMENT",
    4: "LOCA_ERR_UNSUPPORTED_DTYPE", 5: "LOCA_ERR_CUDA", 6: "LOCA_ERR_TIMEOUT",
    7: "LOCA_ERR_WORKSPACE", 8: "LOCA_ERR_UNSUPPORTED", 9: "LOCA_ERR_NUMERIC", 10: "LOCA_ERR_BOUNDS",
}

# (name, restype, argtypes) of every exported entry point
_P = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_F = ctypes.c_float
SIGNATURES = [
    ("loca_version", ctypes.c_int, []),
    ("loca_last_error_string", ctypes.c_char_p, []),
    ("loca_device_status", ctypes.c_int, [ctypes.POINTER(_I32), _P]),
    ("loca_debug_build", ctypes.c_int, []),
    ("loca_set_wait_limit", ctypes.c_int, [ctypes.c_uint64]),
    ("loca_error", ctypes.c_int, [_P, ctypes.c_int, _I64, _I64, _I64, _P, _I32, _P, _P, ctypes.c_int, _P, _P, _P]),
    ("loca_targets_workspace_size", ctypes.c_int, [_I64, _I32, _I64, ctypes.POINTER(_SZ)]),
    ("loca_targets", ctypes.c_int, [_P, _I64, _I32, _P, _P, _I32, _I32, _I64, _P, ctypes.c_int, _P, _P, _SZ, _P]),
    ("loca_accumulate_workspace_size", ctypes.c_int, [_I32, _I64, _I64, ctypes.c_int, ctypes.POINTER(_SZ)]),
    ("loca_accumulate", ctypes.c_int,
     [_P, _P, ctypes.c_int, _I32, _I64, _I64, _P, _F, ctypes.c_int, _P, _P, _P, _P, _SZ, _P]),
    ("loca_accumulate_noalloc", ctypes.c_int,
     [_P, _P, ctypes.c_int, _I32, _I64, _I64, _P, _F, ctypes.c_int, _P, _P, _P, _P]),
    ("loca_accumulate_streamed", ctypes.c_int,
     [_P, _P, _P, ctypes.c_int, _I32, _I64, _I64, _I32, _P, _F, ctypes.c_int, _P, _P, _P, _P, _SZ, _P]),
    ("loca_alignment_workspace_size", ctypes.c_int, [_I64, _I32, _I64, _I32, _I32, ctypes.POINTER(_SZ)]),
    ("loca_alignment", ctypes.c_int, [_P, _P, _I64, _I32, _I64, _I32, _P, _P, _I32, _P, _P, _SZ, _P]),
    ("loca_kspace_workspace_size", ctypes.c_int, [_I32, _I64, _I64, _I32, _I32, _I32, ctypes.POINTER(_SZ)]),
    ("loca_kspace_accumulate", ctypes.c_int,
     [_P, ctypes.c_int, _I32, _I64, _I64, _P, _I32, _P, _I32, _P, _P, _I32, _F, ctypes.c_int, _P, _P, _P, _P, _P,
      _SZ, _P]),
    ("loca_kspace_solve", ctypes.c_int,
     [_P, _P, _P, _P, _P, _P, ctypes.POINTER(_F), _I32, _I32, _I64, _I32, _I32, _I32, _P, _P, _P, _P]),
    ("loca_host_alloc", ctypes.c_int, [_SZ, ctypes.POINTER(ctypes.c_void_p)]),
    ("loca_host_free", ctypes.c_int, [_P]),
    ("loca_batch_step_workspace_size", ctypes.c_int, [_I32, ctypes.POINTER(_SZ)]),
    ("loca_batch_step", ctypes.c_int, [_P, ctypes.c_int, _I32, _I64, _I64, _P, _F, ctypes.c_int, _P, _P, _P, _SZ, _P]),
    ("loca_gram_cross_workspace_size", ctypes.c_int, [ctypes.POINTER(_SZ)]),
    ("loca_gram_cross", ctypes.c_int,
     [_P, _P, ctypes.c_int, _I32, _I64, _I64, _P, ctypes.c_int, _P, _P, _P, _SZ, _P]),
    ("loca_targets_sq_workspace_size", ctypes.c_int, [_I64, _I32, ctypes.POINTER(_SZ)]),
    ("loca_targets_sq", ctypes.c_int, [_P, _I64, _I32, _P, _P, _I32, _I32, _I64, _P, _P, _SZ, _P]),
    ("loca_gram_cross_fused_workspace_size", ctypes.c_int, [_I32, _I64, _I32, ctypes.POINTER(_SZ)]),
    ("loca_gram_cross_fused", ctypes.c_int,
     [_P, ctypes.c_int, _I32, _I64, _I64, _P, _I32, _P, _P, _I32, _P, ctypes.c_int, _P, _P, _P, _SZ, _P]),
    ("loca_ridge_solve_workspace_size", ctypes.c_int, [_I32, _I64, _I32, ctypes.POINTER(_SZ)]),
    ("loca_ridge_solve", ctypes.c_int,
     [_P, _P, _P, _P, _P, _P, ctypes.POINTER(_F), _I32, _I32, _I64, _I32, _P, _P, _P, _P, _P, _SZ, _P]),
    ("loca_step_from_gram", ctypes.c_int, [_P, _I32, _I64, _P, _F, _P, _P, _P]),
    ("loca_calib_fit_workspace_size", ctypes.c_int, [_I64, _I32, _I64, _I32, _I32, ctypes.POINTER(_SZ)]),
    ("loca_calib_fit", ctypes.c_int,
     [_P, _P, _I64, _I32, _I64, _I32, _F, _I32, _P, _P, _P, _P, _SZ, _P]),
    ("loca_calib_fit_rsvd_workspace_size", ctypes.c_int, [_I64, _I32, _I64, _I32, _I32, _I32, ctypes.POINTER(_SZ)]),
    ("loca_calib_fit_rsvd", ctypes.c_int,
     [_P, _P, _I64, _I32, _I64, _I32, _F, _I32, _I32, _I32, _P, _P, _P, _P, _P, _SZ, _P]),
]


class LocaError(RuntimeError):
    def __init__(self, status: int, where: str, message: str):
        self.status = status
        super().__init__(f"{where}: {STATUS_NAMES.get(status, status)}: {message}")


_lib = None
_loaded = {}


def _load(path: str) -> ctypes.CDLL:
    if path not in _loaded:
        if not os.path.exists(path):
            raise RuntimeError(f"{path} is not built: run __graft_entry__.build() (nvcc, sm_103a)")
        h = ctypes.CDLL(path)
        for name, res, args in SIGNATURES:
            fn = getattr(h, name)
            fn.restype = res
            fn.argtypes = args
        _loaded[path] = h
    return _loaded[path]


def lib() -> ctypes.CDLL:
    """The library every function here calls: ``libloca.so`` (built in-tree by
    ``_build.build()``) unless :func:`use_debug_library` switched it; fails loudly if missing."""
    global _lib
    if _lib is None:
        _lib = _load(LIB_PATH)
    return _lib


def use_debug_library(on: bool = True) -> ctypes.CDLL:
    """Route every function of this module to ``libloca_debug.so`` (``_build.build(debug=True)``:
    the same entry points with index bounds checks reported as LOCA_ERR_BOUNDS by
    :func:`loca_device_status`), or back to ``libloca.so``.  Each library keeps its own device
    status word; returns the library now in use."""
    global _lib
    _lib = _load(LIB_DEBUG_PATH if on else LIB_PATH)
    return _lib


def loca_debug_build() -> bool:
    """True when the library in use is the LOCA_DEBUG build."""
    return bool(lib().loca_debug_build())


def _check(rc: int, where: str):
    if rc != 0:
        msg = lib().loca_last_error_string().decode(errors="replace")
        raise LocaError(rc, where, msg)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev(t, name, dtype=None, ndim=None):
    if t is None:
        return
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype not in (dtype if isinstance(dtype, tuple) else (dtype,)):
        raise TypeError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dimensions, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _code(dtype) -> int:
    if dtype == torch.float32:
        return LOCA_F32
    if dtype == torch.bfloat16:
        return LOCA_BF16
    raise TypeError(f"unsupported dtype {dtype}")


def _workspace(nbytes: int, device, given=None):
    if nbytes == 0:
        return None
    if given is not None:
        if given.numel() * given.element_size() < nbytes:
            raise ValueError(f"workspace has {given.numel() * given.element_size()} bytes, need {nbytes}")
        return given
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


def loca_version() -> int:
    return lib().loca_version()


def loca_device_status(stream=None) -> int:
    """Read and clear the device status word (LOCA_OK or a device-side code: LOCA_ERR_TIMEOUT,
    LOCA_ERR_NUMERIC, or in the debug build LOCA_ERR_BOUNDS, whose source line
    :func:`loca_last_error` then names)."""
    out = ctypes.c_int32(0)
    _check(lib().loca_device_status(ctypes.byref(out), _stream(stream)), "loca_device_status")
    return out.value


def loca_last_error() -> str:
    """Message of the last non-OK status of the calling thread (``loca_last_error_string``)."""
    return lib().loca_last_error_string().decode(errors="replace")


def loca_set_wait_limit(ns: int):
    """Test hook: how long a device wait of the tensor-core kernels may take before it
    gives up with LOCA_ERR_TIMEOUT (0 restores the default of 4 s)."""
    _check(lib().loca_set_wait_limit(int(ns)), "loca_set_wait_limit")


def loca_error(logits, label_cols, y, E, w=None, ce=None, normaliser=0, stream=None):
    """Top-layer error at the head: fills ``E`` (N x C float) and optionally ``ce`` (N)."""
    if not isinstance(logits, torch.Tensor) or not logits.is_cuda:
        raise TypeError("logits must be a CUDA tensor")
    if logits.dtype not in (torch.float32, torch.bfloat16):
        raise TypeError(f"logits has dtype {logits.dtype}, expected float32 or bfloat16")
    if logits.dim() != 2 or logits.stride(1) != 1 or logits.stride(0) < logits.shape[1]:
        raise ValueError("logits must be 2-D with unit column stride and row pitch >= V")
    _dev(label_cols, "label_cols", torch.int32, 1)
    _dev(y, "y", torch.int32, 1)
    _dev(E, "E", torch.float32, 2)
    _dev(w, "w", torch.float32, 1)
    _dev(ce, "ce", torch.float32, 1)
    N, V = logits.shape
    C = label_cols.numel()
    if E.shape != (N, C) or y.numel() != N:
        raise ValueError("E must be N x C and y must have N entries")
    rc = lib().loca_error(_ptr(logits), _code(logits.dtype), N, V, logits.stride(0), _ptr(label_cols), C,
                          _ptr(y), _ptr(w), int(normaliser), _ptr(E), _ptr(ce), _stream(stream))
    _check(rc, "loca_error")


def targets_workspace_size(N, L, d) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_targets_workspace_size(N, L, d, ctypes.byref(out)), "loca_targets_workspace_size")
    return out.value


def loca_targets(E, P, Q, T, tsq=None, workspace=None, stream=None):
    """Feedback targets ``T_l = (E P_l) Q_l`` into ``T`` (L x N x d, bf16 or f32) and
    ``tsq`` (L, float64, optional).  A workspace is always used (allocated if not given)."""
    _dev(E, "E", torch.float32, 2)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(T, "T", (torch.float32, torch.bfloat16), 3)
    _dev(tsq, "tsq", torch.float64, 1)
    N, C = E.shape
    L, C2, r = P.shape
    L2, r2, d = Q.shape
    if C2 != C or L2 != L or r2 != r or tuple(T.shape) != (L, N, d):
        raise ValueError("shape mismatch among E (N x C), P (L x C x r), Q (L x r x d), T (L x N x d)")
    nbytes = targets_workspace_size(N, L, d)
    ws = _workspace(nbytes, E.device, workspace)
    rc = lib().loca_targets(_ptr(E), N, C, _ptr(P), _ptr(Q), L, r, d, _ptr(T), _code(T.dtype), _ptr(tsq),
                            _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_targets")


def accumulate_workspace_size(L, N, d, dtype) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_accumulate_workspace_size(L, N, d, _code(dtype), ctypes.byref(out)),
           "loca_accumulate_workspace_size")
    return out.value


def loca_accumulate(X, T, tsq, eta, gram, cross, xsq_total, zero_first, workspace=None, stream=None):
    """Add one mini-batch to the Gram / cross statistics of every block."""
    _dev(X, "X", (torch.float32, torch.bfloat16), 3)
    _dev(T, "T", X.dtype, 3)
    _dev(tsq, "tsq", torch.float64, 1)
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    L, N, d = X.shape
    if tuple(T.shape) != (L, N, d) or tuple(gram.shape) != (L, d, d) or tuple(cross.shape) != (L, d, d):
        raise ValueError("shape mismatch among X, T (L x N x d) and gram, cross (L x d x d)")
    nbytes = accumulate_workspace_size(L, N, d, X.dtype)
    ws = _workspace(nbytes, X.device, workspace)
    rc = lib().loca_accumulate(_ptr(X), _ptr(T), _code(X.dtype), L, N, d, _ptr(tsq), float(eta), int(bool(zero_first)),
                               _ptr(gram), _ptr(cross), _ptr(xsq_total), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_accumulate")


def loca_accumulate_noalloc(X, T, tsq, eta, gram, cross, xsq_total, zero_first, stream=None):
    """loca_accumulate without a workspace, for callers that cannot allocate device memory when
    they call the library; its scratch is a fixed array inside the library (L <= 64 blocks).
    Calls that may overlap on the GPU share that array and must be serialised."""
    _dev(X, "X", (torch.float32, torch.bfloat16), 3)
    _dev(T, "T", X.dtype, 3)
    _dev(tsq, "tsq", torch.float64, 1)
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    L, N, d = X.shape
    if tuple(T.shape) != (L, N, d) or tuple(gram.shape) != (L, d, d) or tuple(cross.shape) != (L, d, d):
        raise ValueError("shape mismatch among X, T (L x N x d) and gram, cross (L x d x d)")
    rc = lib().loca_accumulate_noalloc(_ptr(X), _ptr(T), _code(X.dtype), L, N, d, _ptr(tsq), float(eta),
                                       int(bool(zero_first)), _ptr(gram), _ptr(cross), _ptr(xsq_total),
                                       _stream(stream))
    _check(rc, "loca_accumulate_noalloc")


class _HostBlock:
    """Owns one loca_host_alloc buffer; freed when the last tensor viewing it is gone."""

    def __init__(self, nbytes):
        p = ctypes.c_void_p(0)
        _check(lib().loca_host_alloc(nbytes, ctypes.byref(p)), "loca_host_alloc")
        self.ptr = p.value

    def __del__(self):
        if getattr(self, "ptr", None):
            lib().loca_host_free(ctypes.c_void_p(self.ptr))
            self.ptr = None


def host_empty(shape, dtype):
    """A CPU tensor in loca_host_alloc memory (page-locked, 2 MiB pages, zero-filled): host
    inputs in it copy to the GPU at the full link rate."""
    shape = tuple(int(s) for s in shape)
    n = 1
    for s in shape:
        n *= s
    nbytes = n * torch.empty((), dtype=dtype).element_size()
    if nbytes == 0:
        return torch.empty(shape, dtype=dtype)
    owner = _HostBlock(nbytes)
    buf = (ctypes.c_uint8 * nbytes).from_address(owner.ptr)
    buf.owner = owner  # the tensor keeps `buf` alive, `buf` keeps the allocation
    return torch.frombuffer(buf, dtype=dtype).view(shape)


def loca_accumulate_streamed(X_host, staging, T, tsq, eta, gram, cross, xsq_total, zero_first, group=2,
                             workspace=None, stream=None):
    """loca_accumulate with X in host memory: X_host (L x N x d, CPU tensor, ideally pinned) is
    copied to the device `group` blocks at a time into `staging` (a device tensor with room for
    2 x group x N x d elements, used as two alternating slots) while the statistics of the
    previous group run on the stream."""
    if not isinstance(X_host, torch.Tensor) or X_host.is_cuda or X_host.dim() != 3 or not X_host.is_contiguous():
        raise TypeError("X_host must be a contiguous 3-D CPU tensor")
    _dev(staging, "staging", X_host.dtype)
    _dev(T, "T", X_host.dtype, 3)
    _dev(tsq, "tsq", torch.float64, 1)
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    L, N, d = X_host.shape
    group = max(1, min(int(group), L))
    if tuple(T.shape) != (L, N, d) or tuple(gram.shape) != (L, d, d) or tuple(cross.shape) != (L, d, d):
        raise ValueError("shape mismatch among X_host, T (L x N x d) and gram, cross (L x d x d)")
    if staging.numel() < 2 * group * N * d:
        raise ValueError(f"staging has {staging.numel()} elements, need 2 x group x N x d = {2 * group * N * d}")
    nbytes = accumulate_workspace_size(L, N, d, X_host.dtype)
    ws = _workspace(nbytes, T.device, workspace)
    rc = lib().loca_accumulate_streamed(ctypes.c_void_p(X_host.data_ptr()), _ptr(staging), _ptr(T),
                                        _code(X_host.dtype), L, N, d, group, _ptr(tsq), float(eta),
                                        int(bool(zero_first)), _ptr(gram), _ptr(cross), _ptr(xsq_total),
                                        _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_accumulate_streamed")


def loca_alignment(E_probe, G_probe, P, Q, alpha, workspace=None, stream=None):
    """Per-block cosine between the feedback predictions E P_l Q_l and the probe gradients."""
    _dev(E_probe, "E_probe", torch.float32, 2)
    _dev(G_probe, "G_probe", torch.float32, 3)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(alpha, "alpha", torch.float64, 1)
    Np, m = E_probe.shape
    L, _, d = G_probe.shape
    r = P.shape[2]
    if (tuple(G_probe.shape) != (L, Np, d) or tuple(P.shape) != (L, m, r) or tuple(Q.shape) != (L, r, d)
            or alpha.numel() != L):
        raise ValueError("shape mismatch among E_probe, G_probe, P, Q, alpha")
    out = ctypes.c_size_t(0)
    _check(lib().loca_alignment_workspace_size(Np, m, d, L, r, ctypes.byref(out)), "loca_alignment_workspace_size")
    ws = _workspace(out.value, G_probe.device, workspace)
    rc = lib().loca_alignment(_ptr(E_probe), _ptr(G_probe), Np, m, d, L, _ptr(P), _ptr(Q), r, _ptr(alpha), _ptr(ws),
                              out.value, _stream(stream))
    _check(rc, "loca_alignment")


def kspace_workspace_size(L, N, d, k, C, r) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_kspace_workspace_size(L, N, d, k, C, r, ctypes.byref(out)), "loca_kspace_workspace_size")
    return out.value


def loca_kspace_accumulate(X, A, E, P, Q, eta, G, SC, xsq_total, zero_first, alpha=None, workspace=None,
                           stream=None):
    """The paper's k-space statistics of one mini-batch: G_l (+)= (X_l A_l)^T (X_l A_l),
    SC_l (+)= alpha_l E^T (X_l A_l), xsq_total (+)= ||X_l||^2, with alpha_l = -eta RMS(X_l)/RMS(T_l)
    and T_l = E P_l Q_l never formed."""
    _dev(X, "X", torch.bfloat16, 3)
    _dev(A, "A", torch.float32, 3)
    _dev(E, "E", torch.float32, 2)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(G, "G", torch.float32, 3)
    _dev(SC, "SC", torch.float32, 3)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    _dev(alpha, "alpha", torch.float32, 1)
    L, N, d = X.shape
    k = A.shape[2]
    C, r = P.shape[1], P.shape[2]
    if (tuple(A.shape) != (L, d, k) or tuple(E.shape) != (N, C) or tuple(Q.shape) != (L, r, d)
            or tuple(G.shape) != (L, k, k) or tuple(SC.shape) != (L, C, k) or P.shape[0] != L):
        raise ValueError("shape mismatch among X, A, E, P, Q, G, SC")
    nbytes = kspace_workspace_size(L, N, d, k, C, r)
    ws = _workspace(nbytes, X.device, workspace)
    rc = lib().loca_kspace_accumulate(_ptr(X), LOCA_BF16, L, N, d, _ptr(A), k, _ptr(E), C, _ptr(P), _ptr(Q), r,
                                      float(eta), int(bool(zero_first)), _ptr(G), _ptr(SC), _ptr(xsq_total),
                                      _ptr(alpha), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_kspace_accumulate")


def loca_kspace_solve(G, SC, P, Q, lambda_rel, B, info, xsq_total=None, B_prev=None, C_out=None, stream=None):
    """Ridge solves from the k-space statistics: B[j, l] (G_l + lambda_j I) = C_l with
    C_l = B_prev,l G_l + Q_l^T (P_l^T SC_l); lambda_j = lambda_rel[j] xsq_total[l] / d."""
    _dev(G, "G", torch.float32, 3)
    _dev(SC, "SC", torch.float32, 3)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(B, "B", torch.float32, 4)
    _dev(info, "info", torch.int32, 2)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    _dev(B_prev, "B_prev", torch.float32, 3)
    _dev(C_out, "C_out", torch.float32, 3)
    L, k, _ = G.shape
    C, r = P.shape[1], P.shape[2]
    d = Q.shape[2]
    lam = [float(v) for v in lambda_rel]
    nl = len(lam)
    if tuple(B.shape) != (nl, L, d, k) or tuple(info.shape) != (nl, L) or tuple(SC.shape) != (L, C, k):
        raise ValueError("shape mismatch among G, SC, Q, B, info")
    arr = (ctypes.c_float * nl)(*lam)
    rc = lib().loca_kspace_solve(_ptr(G), _ptr(SC), _ptr(xsq_total), _ptr(P), _ptr(Q), _ptr(B_prev), arr, nl, L, d,
                                 k, C, r, _ptr(B), _ptr(info), _ptr(C_out), _stream(stream))
    _check(rc, "loca_kspace_solve")


def batch_step_workspace_size(L) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_batch_step_workspace_size(L, ctypes.byref(out)), "loca_batch_step_workspace_size")
    return out.value


def loca_batch_step(X, tsq, eta, xsq_total, alpha, zero_first, workspace=None, stream=None):
    """Step of Eq. 10 for one mini-batch: ``alpha[l] = -eta ||X_l|| / sqrt(tsq[l])``; updates
    ``xsq_total``."""
    _dev(X, "X", (torch.float32, torch.bfloat16), 3)
    _dev(tsq, "tsq", torch.float64, 1)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    _dev(alpha, "alpha", torch.float32, 1)
    L, N, d = X.shape
    nbytes = batch_step_workspace_size(L)
    ws = _workspace(nbytes, X.device, workspace)
    rc = lib().loca_batch_step(_ptr(X), _code(X.dtype), L, N, d, _ptr(tsq), float(eta), int(bool(zero_first)),
                               _ptr(xsq_total), _ptr(alpha), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_batch_step")


def gram_cross_workspace_size() -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_gram_cross_workspace_size(ctypes.byref(out)), "loca_gram_cross_workspace_size")
    return out.value


def loca_gram_cross(X, T, alpha, gram, cross, zero_first, workspace=None, stream=None):
    """Statistics of Eq. 9 for one mini-batch with the step ``alpha`` of loca_batch_step."""
    _dev(X, "X", (torch.float32, torch.bfloat16), 3)
    _dev(T, "T", X.dtype, 3)
    _dev(alpha, "alpha", torch.float32, 1)
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    L, N, d = X.shape
    if tuple(T.shape) != (L, N, d) or tuple(gram.shape) != (L, d, d) or tuple(cross.shape) != (L, d, d):
        raise ValueError("shape mismatch among X, T (L x N x d) and gram, cross (L x d x d)")
    nbytes = gram_cross_workspace_size()
    ws = _workspace(nbytes, X.device, workspace)
    rc = lib().loca_gram_cross(_ptr(X), _ptr(T), _code(X.dtype), L, N, d, _ptr(alpha), int(bool(zero_first)),
                               _ptr(gram), _ptr(cross), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_gram_cross")


def targets_sq_workspace_size(N, C) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_targets_sq_workspace_size(N, C, ctypes.byref(out)), "loca_targets_sq_workspace_size")
    return out.value


def loca_targets_sq(E, P, Q, tsq, workspace=None, stream=None):
    """``tsq[l] = ||E P_l Q_l||_F^2`` (float64, L) without forming the targets."""
    _dev(E, "E", torch.float32, 2)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(tsq, "tsq", torch.float64, 1)
    N, C = E.shape
    L, C2, r = P.shape
    L2, r2, d = Q.shape
    if C2 != C or L2 != L or r2 != r or tuple(tsq.shape) != (L,):
        raise ValueError("shape mismatch among E (N x C), P (L x C x r), Q (L x r x d), tsq (L)")
    nbytes = targets_sq_workspace_size(N, C)
    ws = _workspace(nbytes, E.device, workspace)
    rc = lib().loca_targets_sq(_ptr(E), N, C, _ptr(P), _ptr(Q), L, r, d, _ptr(tsq), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_targets_sq")


def gram_cross_fused_workspace_size(L, N, r) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_gram_cross_fused_workspace_size(L, N, r, ctypes.byref(out)),
           "loca_gram_cross_fused_workspace_size")
    return out.value


def loca_gram_cross_fused(X, E, P, Q, alpha, gram, cross, zero_first, workspace=None, stream=None):
    """loca_gram_cross with each block's targets ``T_l = (E P_l) Q_l`` generated inside the kernel."""
    _dev(X, "X", torch.bfloat16, 3)
    _dev(E, "E", torch.float32, 2)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(alpha, "alpha", torch.float32, 1)
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    L, N, d = X.shape
    C, r = P.shape[1], P.shape[2]
    if (tuple(E.shape) != (N, C) or tuple(P.shape) != (L, C, r) or tuple(Q.shape) != (L, r, d)
            or tuple(gram.shape) != (L, d, d) or tuple(cross.shape) != (L, d, d)):
        raise ValueError("shape mismatch among X, E, P, Q, gram, cross")
    nbytes = gram_cross_fused_workspace_size(L, N, r)
    ws = _workspace(nbytes, X.device, workspace)
    rc = lib().loca_gram_cross_fused(_ptr(X), LOCA_BF16, L, N, d, _ptr(E), C, _ptr(P), _ptr(Q), r, _ptr(alpha),
                                     int(bool(zero_first)), _ptr(gram), _ptr(cross), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_gram_cross_fused")


def ridge_solve_workspace_size(L, d, k) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_ridge_solve_workspace_size(L, d, k, ctypes.byref(out)), "loca_ridge_solve_workspace_size")
    return out.value


def loca_ridge_solve(gram, cross, A, lambda_rel, B, info, xsq_total=None, B_prev=None, G_out=None, C_out=None,
                     cross_scale=None, workspace=None, stream=None):
    """Closed-form adapters ``B[j, l] = C_l (G_l + lambda_j I)^-1`` for every block and candidate;
    ``cross_scale`` (L, optional) multiplies ``cross_l``."""
    _dev(gram, "gram", torch.float32, 3)
    _dev(cross, "cross", torch.float32, 3)
    _dev(cross_scale, "cross_scale", torch.float32, 1)
    _dev(A, "A", torch.float32, 3)
    _dev(B, "B", torch.float32, 4)
    _dev(info, "info", torch.int32, 2)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    _dev(B_prev, "B_prev", torch.float32, 3)
    _dev(G_out, "G_out", torch.float32, 3)
    _dev(C_out, "C_out", torch.float32, 3)
    L, d, k = A.shape
    lam = [float(v) for v in lambda_rel]
    nl = len(lam)
    if tuple(B.shape) != (nl, L, d, k) or tuple(info.shape) != (nl, L):
        raise ValueError("B must be nl x L x d x k and info nl x L")
    lam_arr = (ctypes.c_float * max(nl, 1))(*lam)
    nbytes = ridge_solve_workspace_size(L, d, k)
    ws = _workspace(nbytes, A.device, workspace)
    if cross_scale is not None and tuple(cross_scale.shape) != (L,):
        raise ValueError("cross_scale must have L entries")
    rc = lib().loca_ridge_solve(_ptr(gram), _ptr(cross), _ptr(cross_scale), _ptr(xsq_total), _ptr(A), _ptr(B_prev),
                                lam_arr, nl, L, d, k, _ptr(B), _ptr(info), _ptr(G_out), _ptr(C_out), _ptr(ws), nbytes,
                                _stream(stream))
    _check(rc, "loca_ridge_solve")


def loca_step_from_gram(gram, tsq, eta, xsq_total, alpha, stream=None):
    """Step of Eq. 10 for a pass with one mini-batch from ``tr(gram_l) = ||X_l||^2``:
    ``alpha[l] = -eta sqrt(tr(gram_l) / tsq[l])``, ``xsq_total[l] = tr(gram_l)``."""
    _dev(gram, "gram", torch.float32, 3)
    _dev(tsq, "tsq", torch.float64, 1)
    _dev(xsq_total, "xsq_total", torch.float64, 1)
    _dev(alpha, "alpha", torch.float32, 1)
    L, d, d2 = gram.shape
    if d2 != d or tuple(tsq.shape) != (L,) or tuple(xsq_total.shape) != (L,) or tuple(alpha.shape) != (L,):
        raise ValueError("gram must be L x d x d; tsq, xsq_total, alpha must have L entries")
    rc = lib().loca_step_from_gram(_ptr(gram), L, d, _ptr(tsq), float(eta), _ptr(xsq_total), _ptr(alpha),
                                   _stream(stream))
    _check(rc, "loca_step_from_gram")


def calib_fit_workspace_size(Np, m, d, L, r) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_calib_fit_workspace_size(Np, m, d, L, r, ctypes.byref(out)), "loca_calib_fit_workspace_size")
    return out.value


def loca_calib_fit(E_probe, G_probe, beta, r, P, Q, sigma=None, workspace=None, stream=None):
    """Rank-r feedback factors ``P`` (L x m x r), ``Q`` (L x r x d) from probe pairs."""
    _dev(E_probe, "E_probe", torch.float32, 2)
    _dev(G_probe, "G_probe", torch.float32, 3)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(sigma, "sigma", torch.float32, 2)
    Np, m = E_probe.shape
    L, Np2, d = G_probe.shape
    if Np2 != Np or tuple(P.shape) != (L, m, r) or tuple(Q.shape) != (L, r, d):
        raise ValueError("shape mismatch among E_probe, G_probe, P, Q")
    nbytes = calib_fit_workspace_size(Np, m, d, L, r)
    ws = _workspace(nbytes, E_probe.device, workspace)
    rc = lib().loca_calib_fit(_ptr(E_probe), _ptr(G_probe), Np, m, d, L, float(beta), r, _ptr(P), _ptr(Q),
                              _ptr(sigma), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_calib_fit")


def calib_fit_rsvd_workspace_size(Np, m, d, L, r, ell) -> int:
    out = ctypes.c_size_t(0)
    _check(lib().loca_calib_fit_rsvd_workspace_size(Np, m, d, L, r, ell, ctypes.byref(out)),
           "loca_calib_fit_rsvd_workspace_size")
    return out.value


def loca_calib_fit_rsvd(E_probe, G_probe, beta, r, Omega, q, P, Q, sigma=None, workspace=None, stream=None):
    """Rank-r feedback factors for wide error spaces by randomized subspace iteration:
    ``Omega`` (d x ell) is the Gaussian test matrix, ``q`` the number of power iterations."""
    _dev(E_probe, "E_probe", torch.float32, 2)
    _dev(G_probe, "G_probe", torch.float32, 3)
    _dev(Omega, "Omega", torch.float32, 2)
    _dev(P, "P", torch.float32, 3)
    _dev(Q, "Q", torch.float32, 3)
    _dev(sigma, "sigma", torch.float32, 2)
    Np, m = E_probe.shape
    L, Np2, d = G_probe.shape
    ell = Omega.shape[1]
    if (Np2 != Np or Omega.shape[0] != d or tuple(P.shape) != (L, m, r) or tuple(Q.shape) != (L, r, d)
            or (sigma is not None and tuple(sigma.shape) != (L, r))):
        raise ValueError("shape mismatch among E_probe, G_probe, Omega, P, Q, sigma")
    nbytes = calib_fit_rsvd_workspace_size(Np, m, d, L, r, ell)
    ws = _workspace(nbytes, E_probe.device, workspace)
    rc = lib().loca_calib_fit_rsvd(_ptr(E_probe), _ptr(G_probe), Np, m, d, L, float(beta), r, ell, int(q),
                                   _ptr(Omega), _ptr(P), _ptr(Q), _ptr(sigma), _ptr(ws), nbytes, _stream(stream))
    _check(rc, "loca_calib_fit_rsvd")


class Pass:
    """Device buffers and workspaces for repeated Stage-II outer iterations of one shape.

    ``run()`` enqueues loca_error -> (loca_targets -> loca_accumulate per mini-batch) ->
    loca_ridge_solve on the current stream and allocates nothing.
    """

    def __init__(self, L, N, d, C, r, k, act_dtype, lambda_rel, eta, micro_batches=1, device="cuda",
                 t_dtype=None):
        self.L, self.N, self.d, self.C, self.r, self.k = L, N, d, C, r, k
        self.eta = float(eta)
        self.lambda_rel = [float(v) for v in lambda_rel]
        self.mb = int(micro_batches)
        self.nb = -(-N // self.mb)
        dev = torch.device(device)
        t_dtype = act_dtype if t_dtype is None else t_dtype
        f32 = dict(dtype=torch.float32, device=dev)
        self.E = torch.empty((N, C), **f32)
        self.ce = torch.empty((N,), **f32)
        self.T = torch.empty((L, self.nb, d), dtype=t_dtype, device=dev)
        self.tsq = torch.empty((L,), dtype=torch.float64, device=dev)
        self.gram = torch.empty((L, d, d), **f32)
        self.cross = torch.empty((L, d, d), **f32)
        self.xsq = torch.empty((L,), dtype=torch.float64, device=dev)
        nl = len(self.lambda_rel)
        self.B = torch.empty((nl, L, d, k), **f32)
        self.info = torch.empty((nl, L), dtype=torch.int32, device=dev)
        self.ws_t = _workspace(targets_workspace_size(self.nb, L, d), dev)
        self.ws_a = _workspace(accumulate_workspace_size(L, self.nb, d, act_dtype), dev)
        self.ws_s = _workspace(ridge_solve_workspace_size(L, d, k), dev)

    def run(self, logits, label_cols, y, X, P, Q, A, B_prev=None, normaliser=0, stream=None):
        """``X``: one ``L x N x d`` tensor, or a list of per-mini-batch ``L x N_m x d`` tensors
        (contiguous token ranges of ``ceil(N / micro_batches)`` tokens, in order)."""
        loca_error(logits, label_cols, y, self.E, ce=self.ce, normaliser=normaliser, stream=stream)
        batches = X if isinstance(X, (list, tuple)) else [X]
        if len(batches) != self.mb:
            raise ValueError(f"expected {self.mb} mini-batches of X, got {len(batches)}")
        n0 = 0
        for m, Xm in enumerate(batches):
            nm = Xm.shape[1]
            Tm = self.T.view(-1)[: self.L * nm * self.d].view(self.L, nm, self.d)
            loca_targets(self.E[n0:n0 + nm], P, Q, Tm, tsq=self.tsq, workspace=self.ws_t, stream=stream)
            loca_accumulate(Xm, Tm, self.tsq, self.eta, self.gram, self.cross, self.xsq, zero_first=(m == 0),
                            workspace=self.ws_a, stream=stream)
            n0 += nm
        if n0 != self.N:
            raise ValueError(f"mini-batches hold {n0} tokens, expected {self.N}")
        loca_ridge_solve(self.gram, self.cross, A, self.lambda_rel, self.B, self.info, xsq_total=self.xsq,
                         B_prev=B_prev, workspace=self.ws_s, stream=stream)
        return self.B
