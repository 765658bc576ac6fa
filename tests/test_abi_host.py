"""Host-side checks of the C ABI (no GPU needed): the library builds and loads, exports every
symbol ``include/loca.h`` declares, the binding knows every one of them, and argument
validation rejects bad calls with the documented status codes before any CUDA call."""

import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "loca.h")


def _declared():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(loca_[a-z0-9_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def L():
    from paper_2608_03020_gb300 import _build
    from paper_2608_03020_gb300 import loca

    _build.build()
    return loca.lib()


def test_header_declares_the_five_hot_path_calls():
    names = _declared()
    for n in ("loca_calib_fit", "loca_error", "loca_targets", "loca_accumulate", "loca_ridge_solve"):
        assert n in names


def test_library_exports_every_declared_symbol(L):
    for name in _declared():
        assert hasattr(L, name), name


def test_binding_covers_every_declared_symbol():
    from paper_2608_03020_gb300 import loca

    assert sorted(n for n, _, _ in loca.SIGNATURES) == _declared()


def test_version(L):
    assert L.loca_version() == 100


def _ws(fn, *args):
    out = ctypes.c_size_t(0)
    rc = fn(*args, ctypes.byref(out))
    return rc, out.value


def test_workspace_sizes(L):
    rc, n = _ws(L.loca_targets_workspace_size, 131072, 28, 3584)
    assert rc == 0 and n >= 8 * 28 * 14 * (131072 // 4096) * 4 + 4 and n % 256 == 0
    rc, n = _ws(L.loca_accumulate_workspace_size, 28, 131072, 3584, 1)
    assert rc == 0 and n > 0
    rc, n = _ws(L.loca_ridge_solve_workspace_size, 28, 3584, 16)
    assert rc == 0 and n >= 2 * 4 * 28 * 3584 * 16
    rc, _ = _ws(L.loca_ridge_solve_workspace_size, 0, 3584, 16)
    assert rc == 2  # LOCA_ERR_SHAPE
    assert L.loca_targets_workspace_size(1, 1, 1, None) == 1  # NULL out pointer


def test_validation_codes(L):
    # every call below is rejected on the host before any CUDA call
    P = ctypes.c_void_p
    fake = P(256)  # never dereferenced: validation fails first
    # bad dtype code
    assert L.loca_error(fake, 7, 4, 4, 4, fake, 4, fake, None, 0, fake, None, None) == 4
    # C > V
    assert L.loca_error(fake, 0, 4, 4, 4, fake, 5, fake, None, 0, fake, None, None) == 2
    # normaliser out of range
    assert L.loca_error(fake, 0, 4, 4, 4, fake, 4, fake, None, 2, fake, None, None) == 1
    # missing E
    assert L.loca_error(fake, 0, 4, 4, 4, fake, 4, fake, None, 0, None, None, None) == 1
    # N == 0 is a no-op
    assert L.loca_error(None, 0, 0, 4, 4, None, 4, None, None, 0, None, None, None) == 0
    msg = L.loca_last_error_string()
    assert msg == b""
    # r out of range
    assert L.loca_targets(fake, 8, 4, fake, fake, 2, 33, 64, fake, 1, None, fake, 1 << 20, None) == 2
    # misaligned T (T must be 16-byte aligned)
    assert L.loca_targets(fake, 8, 4, fake, fake, 2, 4, 64, P(258), 1, None, fake, 1 << 20, None) == 3
    # no workspace
    assert L.loca_targets(fake, 8, 4, fake, fake, 2, 4, 64, fake, 1, fake, None, 0, None) == 7
    # bf16 statistics need d % 8 == 0
    assert L.loca_accumulate(fake, fake, 1, 2, 64, 60, fake, ctypes.c_float(0.01), 1, fake, fake, fake,
                             fake, 1 << 20, None) == 2
    # negative eta
    assert L.loca_accumulate(fake, fake, 1, 2, 64, 64, fake, ctypes.c_float(-1.0), 1, fake, fake, fake,
                             fake, 1 << 20, None) == 1
    # workspace too small
    assert L.loca_accumulate(fake, fake, 1, 2, 64, 64, fake, ctypes.c_float(0.01), 1, fake, fake, fake,
                             fake, 16, None) == 7
    assert b"workspace" in L.loca_last_error_string()
    # lambda_rel must be positive
    lam = (ctypes.c_float * 2)(1e-3, 0.0)
    assert L.loca_ridge_solve(fake, fake, None, None, fake, None, lam, 2, 2, 64, 4, fake, fake, None, None,
                              fake, 1 << 24, None) == 1
    # k above the supported maximum
    lam = (ctypes.c_float * 1)(1e-3)
    assert L.loca_ridge_solve(fake, fake, None, None, fake, None, lam, 1, 2, 64, 33, fake, fake, None, None,
                              fake, 1 << 24, None) == 2
    # step from the Gram trace: L out of range, missing tsq
    assert L.loca_step_from_gram(fake, 0, 64, fake, ctypes.c_float(0.01), fake, fake, None) == 2
    assert L.loca_step_from_gram(fake, 2, 64, None, ctypes.c_float(0.01), fake, fake, None) == 1
    # streamed accumulate: group < 1, missing host X
    assert L.loca_accumulate_streamed(fake, fake, fake, 1, 2, 64, 64, 0, fake, ctypes.c_float(0.01), 1, fake,
                                      fake, fake, fake, 1 << 20, None) == 2
    assert L.loca_accumulate_streamed(None, fake, fake, 1, 2, 64, 64, 1, fake, ctypes.c_float(0.01), 1, fake,
                                      fake, fake, fake, 1 << 20, None) == 1
    # k-space path: bf16 only, C and r limits, d % 8
    assert L.loca_kspace_accumulate(fake, 0, 2, 64, 64, fake, 4, fake, 2, fake, fake, 4, ctypes.c_float(0.01), 1,
                                    fake, fake, fake, None, fake, 1 << 20, None) == 4
    assert L.loca_kspace_accumulate(fake, 1, 2, 64, 64, fake, 4, fake, 17, fake, fake, 4, ctypes.c_float(0.01), 1,
                                    fake, fake, fake, None, fake, 1 << 20, None) == 2
    assert L.loca_kspace_accumulate(fake, 1, 2, 64, 60, fake, 4, fake, 2, fake, fake, 4, ctypes.c_float(0.01), 1,
                                    fake, fake, fake, None, fake, 1 << 20, None) == 2
    lam = (ctypes.c_float * 1)(1e-3)
    assert L.loca_kspace_solve(fake, fake, None, fake, fake, None, lam, 1, 2, 64, 4, 2, 33, fake, fake, None,
                               None) == 2
    rc, n = _ws(L.loca_kspace_workspace_size, 28, 131072, 3584, 16, 4, 16)
    rc2, n2 = _ws(L.loca_kspace_workspace_size, 28, 1024, 3584, 16, 4, 16)
    # W_l (2 x 16 x d bf16 per block) plus partial slots; only the tiny E^T E partials grow with N
    assert rc == 0 and rc2 == 0 and n2 <= n < n2 + (1 << 21) and n >= 28 * 32 * 3584 * 2
    # fused targets: bf16 X only, r and C limits, misaligned gram, missing E; ||T||^2 limits
    f = ctypes.c_float
    assert L.loca_gram_cross_fused(fake, 0, 2, 64, 64, fake, 4, fake, fake, 16, fake, 1, fake, fake, fake,
                                   1 << 20, None) == 4
    assert L.loca_gram_cross_fused(fake, 1, 2, 64, 64, fake, 4, fake, fake, 33, fake, 1, fake, fake, fake,
                                   1 << 20, None) == 2
    assert L.loca_gram_cross_fused(fake, 1, 2, 64, 64, fake, 65, fake, fake, 16, fake, 1, fake, fake, fake,
                                   1 << 20, None) == 2
    assert L.loca_gram_cross_fused(fake, 1, 2, 64, 64, fake, 4, fake, fake, 16, fake, 1, P(260), fake, fake,
                                   1 << 20, None) == 3
    assert L.loca_gram_cross_fused(fake, 1, 2, 64, 64, None, 4, fake, fake, 16, fake, 1, fake, fake, fake,
                                   1 << 20, None) == 1
    assert L.loca_gram_cross_fused(fake, 1, 2, 64, 64, fake, 4, fake, fake, 16, fake, 1, fake, fake, fake,
                                   8, None) == 7
    assert L.loca_targets_sq(fake, 64, 4, fake, fake, 2, 33, 64, fake, fake, 1 << 20, None) == 2
    assert L.loca_targets_sq(fake, 64, 4, fake, fake, 2, 8, 64, None, fake, 1 << 20, None) == 1
    assert L.loca_targets_sq(fake, 64, 4, fake, fake, 2, 8, 64, fake, fake, 8, None) == 7
    rc, n = _ws(L.loca_gram_cross_fused_workspace_size, 28, 131072, 16)
    assert rc == 0 and n >= 256 + 4 * 28 * 131072 * 16
    rc, _ = _ws(L.loca_gram_cross_fused_workspace_size, 28, 131072, 33)
    assert rc == 2
    rc, n = _ws(L.loca_targets_sq_workspace_size, 131072, 4)
    assert rc == 0 and n >= 8 * 16 * (131072 // 2048) and n % 256 == 0
    del f
    # host memory: freeing NULL is a no-op; a pointer the library did not hand out is rejected
    assert L.loca_host_free(None) == 0
    assert L.loca_host_free(fake) == 1
    # calibration: r > m
    assert L.loca_calib_fit(fake, fake, 16, 4, 64, 2, ctypes.c_float(0.1), 5, fake, fake, None, fake,
                            1 << 20, None) == 2
    # calibration: beta <= 0
    assert L.loca_calib_fit(fake, fake, 16, 4, 64, 2, ctypes.c_float(0.0), 2, fake, fake, None, fake,
                            1 << 20, None) == 1


def test_calib_rsvd_validation(L):
    fake = ctypes.c_void_p(256)
    f = ctypes.c_float

    def call(Np=64, m=128, d=96, Lb=2, beta=0.1, r=4, ell=8, q=1, omega=fake, ws_bytes=1 << 40):
        return L.loca_calib_fit_rsvd(fake, fake, Np, m, d, Lb, f(beta), r, ell, q, omega, fake, fake, None, fake,
                                     ws_bytes, None)

    assert call(r=9) == 2            # r > ell
    assert call(ell=65, r=4) == 2    # ell above the limit
    assert call(m=4) == 2            # m < ell
    assert call(d=4) == 2            # d < ell
    assert call(m=16385) == 2        # m above the fp64 vector limit
    assert call(Np=0) == 2
    assert call(Np=65535 * 64 + 1) == 2
    assert call(q=17) == 1
    assert call(q=-1) == 1
    assert call(beta=0.0) == 1
    assert call(omega=None) == 1
    assert call(ws_bytes=16) == 7    # workspace smaller than required
    rc, n = _ws(L.loca_calib_fit_rsvd_workspace_size, 8192, 3584, 3584, 28, 16, 32)
    # E^T E (m x m fp64) and its fp32 copy, plus the ell-column blocks of every block (two
    # m-wide fp64 and one fp32, one d-wide fp64 and its fp32 copy, one Np-wide fp32) dominate
    n_cols = 28 * 32
    floor = 12 * 3584 * 3584 + (8 * 2 * 3584 + 4 * 3584 + 12 * 3584 + 4 * 8192) * n_cols
    assert rc == 0 and floor <= n < floor + (16 << 20) and n % 256 == 0
    assert _ws(L.loca_calib_fit_rsvd_workspace_size, 8192, 3584, 3584, 28, 33, 32)[0] == 2


def test_debug_library_builds_and_exports_every_declared_symbol(L):
    """The LOCA_DEBUG build (bounds checks in every kernel) has the release library's ABI and says
    which it is; the release build compiles the checks away."""
    from paper_2608_03020_gb300 import _build
    from paper_2608_03020_gb300 import loca

    _build.build(debug=True)
    D = loca.use_debug_library(True)
    try:
        for name in _declared():
            assert hasattr(D, name), name
        assert loca.loca_debug_build() and D.loca_version() == L.loca_version()
    finally:
        loca.use_debug_library(False)
    assert not loca.loca_debug_build()
    # host validation is the same code in both builds
    assert D.loca_targets_workspace_size(1, 1, 1, None) == 1
