"""The LOCA_DEBUG build (``libloca_debug.so``) on the GPU.

Every kernel of that build checks the index of each global access it computes against the
extent the sizes of the call give, skips a failing access and records LOCA_ERR_BOUNDS (no trap).
Here the whole pass of the tiny and the Qwen2.5-0.5B workloads, and the k-space path, the
fused-targets statistics, the alignment diagnostic and both calibration fits at small sizes, run
through it with every output and workspace buffer placed between two poisoned guard bands; after
each call the guards must be intact and the status word clear, and the results must equal the
release library's on the same inputs.  A last test feeds a label column outside the logit row:
the debug build's check turns it into LOCA_ERR_BOUNDS at the line of the head-error kernel, with
the read skipped (that input is never given to the release build, which does not check it).
"""

import ctypes

import numpy as np
import pytest
import torch

from synth import inputs as S

pytestmark = pytest.mark.gpu

GUARD = 16384  # bytes of poison on each side of a buffer
POISON = 0xA5


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    _build.build(debug=True)
    from paper_2608_03020_gb300 import loca

    loca.use_debug_library(False)
    yield loca
    loca.use_debug_library(False)


class Guarded:
    """Device buffers of the pass, each inside a poisoned byte band on both sides; ``check``
    also reads the library's status word."""

    def __init__(self, lc):
        self.lc = lc
        self.bufs = []

    def empty(self, shape, dtype):
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        raw = torch.full((n + 2 * GUARD,), POISON, dtype=torch.uint8, device="cuda")
        self.bufs.append((raw, n))
        mid = raw[GUARD:GUARD + n]
        return mid.view(dtype).view(shape) if n else torch.empty(shape, dtype=dtype, device="cuda")

    def workspace(self, nbytes):
        return self.empty((max(int(nbytes), 1),), torch.uint8)

    def check(self, where):
        torch.cuda.synchronize()
        for i, (raw, n) in enumerate(self.bufs):
            head = raw[:GUARD]
            tail = raw[GUARD + n:]
            assert bool((head == POISON).all()) and bool((tail == POISON).all()), f"{where}: guard of buffer {i} written"
        _status(self.lc, where)


def _status(lc, where):
    st = lc.loca_device_status()
    assert st == 0, f"{where}: device status {st}: {lc.loca_last_error()}"


def _rel(a, b):
    a = a.detach().double().cpu()
    b = b.detach().double().cpu()
    return float((a - b).norm() / max(float(b.norm()), 1e-300))


def _pass(lc, w, inp, mk):
    """Every statistics and solve call of one pass on the workload's inputs; outputs and
    workspaces from ``mk`` (a Guarded, which checks its bands after each call, or plain)."""
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, k, r = w.L, w.N, w.d, w.C, w.k, w.r
    nl = len(w.lambda_rel)
    f32, f64 = torch.float32, torch.float64
    bf16 = X.dtype == torch.bfloat16
    chk = getattr(mk, "check", lambda where: torch.cuda.synchronize())
    o = {}
    o["E"], o["ce"] = mk.empty((N, C), f32), mk.empty((N,), f32)
    lc.loca_error(z, cols, y, o["E"], ce=o["ce"])
    chk("loca_error")
    o["T"], o["tsq"] = mk.empty((L, N, d), X.dtype), mk.empty((L,), f64)
    lc.loca_targets(o["E"], P, Q, o["T"], tsq=o["tsq"], workspace=mk.workspace(lc.targets_workspace_size(N, L, d)))
    chk("loca_targets")
    o["gram"], o["cross"] = mk.empty((L, d, d), f32), mk.empty((L, d, d), f32)
    ones = torch.ones((L,), dtype=f32, device="cuda")
    lc.loca_gram_cross(X, o["T"], ones, o["gram"], o["cross"], zero_first=True,
                       workspace=mk.workspace(lc.gram_cross_workspace_size()))
    chk("loca_gram_cross")
    o["xsq"], o["alpha"] = mk.empty((L,), f64), mk.empty((L,), f32)
    lc.loca_step_from_gram(o["gram"], o["tsq"], w.eta, o["xsq"], o["alpha"])
    chk("loca_step_from_gram")
    o["B"], o["info"] = mk.empty((nl, L, d, k), f32), mk.empty((nl, L), torch.int32)
    o["G_out"], o["C_out"] = mk.empty((L, k, k), f32), mk.empty((L, d, k), f32)
    lc.loca_ridge_solve(o["gram"], o["cross"], A, w.lambda_rel, o["B"], o["info"], xsq_total=o["xsq"],
                        G_out=o["G_out"], C_out=o["C_out"], cross_scale=o["alpha"],
                        workspace=mk.workspace(lc.ridge_solve_workspace_size(L, d, k)))
    chk("loca_ridge_solve")
    o["xsq2"], o["alpha2"] = mk.empty((L,), f64), mk.empty((L,), f32)
    lc.loca_batch_step(X, o["tsq"], w.eta, o["xsq2"], o["alpha2"], zero_first=True,
                       workspace=mk.workspace(lc.batch_step_workspace_size(L)))
    chk("loca_batch_step")
    o["gram2"], o["cross2"], o["xsq3"] = mk.empty((L, d, d), f32), mk.empty((L, d, d), f32), mk.empty((L,), f64)
    lc.loca_accumulate(X, o["T"], o["tsq"], w.eta, o["gram2"], o["cross2"], o["xsq3"], zero_first=True,
                       workspace=mk.workspace(lc.accumulate_workspace_size(L, N, d, X.dtype)))
    chk("loca_accumulate")
    o["tsq2"] = mk.empty((L,), f64)
    lc.loca_targets_sq(o["E"], P, Q, o["tsq2"], workspace=mk.workspace(lc.targets_sq_workspace_size(N, C)))
    chk("loca_targets_sq")
    if bf16:
        o["G"], o["SC"] = mk.empty((L, k, k), f32), mk.empty((L, C, k), f32)
        o["xsq4"], o["alpha4"] = mk.empty((L,), f64), mk.empty((L,), f32)
        lc.loca_kspace_accumulate(X, A, o["E"], P, Q, w.eta, o["G"], o["SC"], o["xsq4"], zero_first=True,
                                  alpha=o["alpha4"], workspace=mk.workspace(lc.kspace_workspace_size(L, N, d, k, C, r)))
        chk("loca_kspace_accumulate")
        o["Bk"], o["infok"], o["Ck"] = mk.empty((nl, L, d, k), f32), mk.empty((nl, L), torch.int32), mk.empty((L, d, k), f32)
        lc.loca_kspace_solve(o["G"], o["SC"], P, Q, w.lambda_rel, o["Bk"], o["infok"], xsq_total=o["xsq4"], C_out=o["Ck"])
        chk("loca_kspace_solve")
        o["gram3"], o["cross3"] = mk.empty((L, d, d), f32), mk.empty((L, d, d), f32)
        lc.loca_gram_cross_fused(X, o["E"], P, Q, ones, o["gram3"], o["cross3"], zero_first=True,
                                 workspace=mk.workspace(lc.gram_cross_fused_workspace_size(L, N, r)))
        chk("loca_gram_cross_fused")
    torch.cuda.synchronize()
    return o


class Plain:
    @staticmethod
    def empty(shape, dtype):
        return torch.empty(shape, dtype=dtype, device="cuda")

    @staticmethod
    def workspace(nbytes):
        return torch.empty((max(int(nbytes), 1),), dtype=torch.uint8, device="cuda")


def _compare(ref, got, where):
    for key, a in ref.items():
        b = got[key]
        if a.dtype == torch.int32:
            assert torch.equal(a, b), f"{where}: {key}"
        else:
            rel = _rel(b, a)
            assert rel <= 1e-6, f"{where}: {key} differs from the release build by {rel:.2e}"


@pytest.mark.parametrize("name", ["tiny", "qwen2.5-0.5b"])
def test_debug_build_pass_keeps_every_access_inside_its_buffer(lc, name):
    w = S.WORKLOADS[name]
    inp = S.device_inputs(w, seed=3, device="cuda")
    ref = _pass(lc, w, inp, Plain)
    _status(lc, "release pass")
    try:
        lc.use_debug_library(True)
        assert lc.loca_debug_build()
        got = _pass(lc, w, inp, Guarded(lc))
    finally:
        lc.use_debug_library(False)
    assert int(got["info"].abs().sum()) == 0
    _compare(ref, got, name)
    del ref, got, inp
    torch.cuda.empty_cache()


def _calib(lc, mk, pp, pw, L, r, beta, Om, q):
    chk = getattr(mk, "check", lambda where: torch.cuda.synchronize())
    E, G = pp["E_probe"], pp["G_probe"]
    Np, m = E.shape
    d = G.shape[2]
    o = {}
    o["P"], o["Q"], o["sig"] = mk.empty((L, m, r), torch.float32), mk.empty((L, r, d), torch.float32), mk.empty((L, r), torch.float32)
    lc.loca_calib_fit(E, G, beta, r, o["P"], o["Q"], sigma=o["sig"],
                      workspace=mk.workspace(lc.calib_fit_workspace_size(Np, m, d, L, r)))
    chk("loca_calib_fit")
    o["align"] = mk.empty((L,), torch.float64)
    n_al = ctypes.c_size_t(0)
    assert lc.lib().loca_alignment_workspace_size(Np, m, d, L, r, ctypes.byref(n_al)) == 0
    lc.loca_alignment(E, G, o["P"], o["Q"], o["align"], workspace=mk.workspace(n_al.value))
    chk("loca_alignment")
    Ew, Gw = pw["E_probe"], pw["G_probe"]
    Npw, mw = Ew.shape
    dw = Gw.shape[2]
    ell = Om.shape[1]
    o["Pw"], o["Qw"], o["sigw"] = (mk.empty((L, mw, r), torch.float32), mk.empty((L, r, dw), torch.float32),
                                   mk.empty((L, r), torch.float32))
    lc.loca_calib_fit_rsvd(Ew, Gw, beta, r, Om, q, o["Pw"], o["Qw"], sigma=o["sigw"],
                           workspace=mk.workspace(lc.calib_fit_rsvd_workspace_size(Npw, mw, dw, L, r, ell)))
    chk("loca_calib_fit_rsvd")
    torch.cuda.synchronize()
    return o


def test_debug_build_calibration_and_alignment_keep_every_access_inside_its_buffer(lc):
    L, r = 3, 4
    pp = S.device_probe_pairs(2000, 4, 300, L, rank=4, seed=5)
    pw = S.device_probe_pairs(1500, 200, 200, L, rank=r, seed=6)
    Om = torch.from_numpy(S.omega_matrix(200, 12, seed=6)).cuda()
    args = (pp, pw, L, r, 0.05, Om, 2)
    ref = _calib(lc, Plain, *args)
    _status(lc, "release calibration")
    try:
        lc.use_debug_library(True)
        got = _calib(lc, Guarded(lc), *args)
    finally:
        lc.use_debug_library(False)
    _compare(ref, got, "calibration")


def test_debug_build_reports_a_label_column_outside_the_row(lc):
    """A label column >= V (device data the host cannot check): the debug build's check skips the
    read, records LOCA_ERR_BOUNDS at the head-error kernel's line and the next read is clear."""
    w = S.WORKLOADS["tiny"]
    inp = S.device_inputs(w, seed=1, device="cuda")
    cols = inp["label_cols"].clone()
    cols[1] = w.V + 5
    try:
        lc.use_debug_library(True)
        assert lc.loca_debug_build()  # this input goes to the checked build only
        g = Guarded(lc)
        E, ce = g.empty((w.N, w.C), torch.float32), g.empty((w.N,), torch.float32)
        lc.loca_error(inp["z"], cols, inp["y"], E, ce=ce)
        torch.cuda.synchronize()
        st = lc.loca_device_status()
        msg = lc.loca_last_error()
        assert st == 10, (st, msg)  # LOCA_ERR_BOUNDS
        assert "error.cu:" in msg, msg
        assert lc.loca_device_status() == 0
        g.check("loca_error with a bad column")
        # the column that was in range still gives its error entries
        assert bool(torch.isfinite(E[:, 0]).all())
    finally:
        lc.use_debug_library(False)
