"""GPU parity of the randomized rank-r feedback fit for wide error spaces (Eq. 5; S5; the
paper's m = d form) against the fp64 oracle's calib_fit_rsvd on the same test matrix, and
against the exact truncated SVD (calib_fit) where the spectrum has a gap.

Tolerance: as for loca_calib_fit, the products with E and G_l come from fp32 products summed
in fp32 over 128-term runs and in fp64 across runs (relative error ~1e-7, times the condition
number of E^T E + beta I in the solves); the factorisation, solves, bases and the
Rayleigh-Ritz step run in fp64.  The rank-r map P Q and each factor are within 1e-5 relative
Frobenius (the fp32-input tolerance; measured 1.3e-7 to 6.2e-7) when the retained singular
values are separated from the rest (planted rank r); the worst-case envelope of the arithmetic
(``pq_bound``) is printed beside each error.  Singular values are Weyl-stable (no gap needed)
and match to 1e-5 of sigma_1.
"""

import numpy as np
import pytest
import torch

from oracle import loca_oracle as O
from test_calib_gpu import pq_bound
from synth import inputs as S

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    from paper_2608_03020_gb300 import loca

    loca.lib()
    return loca


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


def _dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


def _fit(lc, E, G, beta, r, Om, q):
    L, Np, d = G.shape
    m = E.shape[1]
    P = torch.full((L, m, r), 7.0, device="cuda")
    Q = torch.full((L, r, d), 7.0, device="cuda")
    sig = torch.full((L, r), 7.0, device="cuda")
    lc.loca_device_status()
    lc.loca_calib_fit_rsvd(E, G, beta, r, Om, q, P, Q, sigma=sig)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    return P.cpu().numpy().astype(np.float64), Q.cpu().numpy().astype(np.float64), sig.cpu().numpy().astype(np.float64)


def _beta(E):
    E64 = np.asarray(E, np.float64)
    return 1e-3 * float(np.sum(E64 * E64)) / E64.shape[1]


# Np, m, d, L, planted rank, r, ell, q, anisotropic E
CASES = [
    (1024, 200, 300, 2, 4, 4, 12, 2, True),   # m, d not multiples of 64
    (1000, 130, 70, 3, 8, 8, 16, 1, False),   # ragged Np; ell = 16 instance
    (700, 96, 128, 1, 6, 6, 40, 0, True),     # ell = 64 instance, no power iteration
    (600, 64, 64, 2, 5, 5, 32, 2, True),      # exact tiles; ell = 32 instance
    (2048, 1024, 1024, 2, 8, 8, 16, 2, True),  # wide error space, m = d
]


@pytest.mark.parametrize("Np,m,d,L,rank,r,ell,q,esc", CASES)
def test_rsvd_parity(lc, Np, m, d, L, rank, r, ell, q, esc):
    pp = S.host_probe_pairs(Np=Np, m=m, d=d, L=L, rank=rank, seed=Np + m + d, e_scales=esc)
    E, G = pp["E_probe"], pp["G_probe"]
    Om = S.omega_matrix(d, ell, seed=m + d)
    beta = _beta(E)
    P, Q, sig = _fit(lc, _dev(E), _dev(G), beta, r, _dev(Om), q)
    Pr, Qr, sr = O.calib_fit_rsvd(E, G, beta, r, Om, q)
    _, _, _, Fh = O.calib_fit(E, G, beta, r)
    for l in range(L):
        err = _rel(P[l] @ Q[l], Pr[l] @ Qr[l])
        print(f"block {l}: P Q rel err {err:.2e} (worst-case bound of the exact fit's arithmetic "
              f"{pq_bound(E, beta, Fh[l], r):.2e})")
        # the fp32-input tolerance: measured 1.3e-7 to 6.2e-7 (fp32 power iterations and GEMM
        # operands, fp64 for the last solve and the Rayleigh-Ritz step)
        assert err < 1e-5, l
        assert np.max(np.abs(sig[l] - sr[l])) < 1e-5 * sr[l, 0], (sig[l], sr[l])
        print(f"block {l}: factor rel err Q {_rel(Q[l], Qr[l]):.2e} P {_rel(P[l], Pr[l]):.2e}")
        assert _rel(Q[l], Qr[l]) < 1e-5 and _rel(P[l], Pr[l]) < 1e-5, l
        assert np.allclose(Q[l] @ Q[l].T, np.eye(r), atol=1e-5)
    if q >= 1:
        # gapped spectrum: the randomized fit is the exact truncated SVD to rounding
        Pe, Qe, se, _ = O.calib_fit(E, G, beta, r)
        for l in range(L):
            assert _rel(P[l] @ Q[l], Pe[l] @ Qe[l]) < 1e-4, l
            assert np.max(np.abs(sig[l] - se[l])) < 1e-5 * se[l, 0]


def test_rsvd_noise_bulk_singular_values(lc):
    """r beyond the planted rank: the trailing retained directions sit in the noise bulk, where
    the rank-r map is not well conditioned, but the Ritz values are (Weyl); they match the
    oracle's on the same test matrix and lie below the exact singular values."""
    Np, m, d, L = 1500, 160, 200, 2
    pp = S.host_probe_pairs(Np=Np, m=m, d=d, L=L, rank=3, seed=5, e_scales=True)
    E, G = pp["E_probe"], pp["G_probe"]
    r, ell, q = 10, 24, 2
    Om = S.omega_matrix(d, ell, seed=6)
    beta = _beta(E)
    P, Q, sig = _fit(lc, _dev(E), _dev(G), beta, r, _dev(Om), q)
    _, _, sr = O.calib_fit_rsvd(E, G, beta, r, Om, q)
    _, _, se, Fh = O.calib_fit(E, G, beta, r)
    for l in range(L):
        assert np.max(np.abs(sig[l] - sr[l])) < 1e-5 * sr[l, 0]
        assert np.all(sig[l] <= se[l] * (1 + 1e-5))
        assert np.allclose(Q[l] @ Q[l].T, np.eye(r), atol=1e-5)
        # the top 3 (gapped) directions agree with the exact fit
        assert _rel(P[l, :, :3] @ Q[l, :3], _top(Fh[l], 3)) < 1e-4


def _top(F, k):
    U, s, Vt = np.linalg.svd(F, full_matrices=False)
    return (U[:, :k] * s[:k]) @ Vt[:k]


def test_rsvd_full_width_equals_exact_gpu_fit(lc):
    """ell = m: the sketch spans the error space and the randomized fit equals the exact GPU
    fit (loca_calib_fit) of the same pairs."""
    pp = S.host_probe_pairs(Np=900, m=24, d=150, L=2, rank=24, noise=0.3, seed=8)
    E, G = _dev(pp["E_probe"]), _dev(pp["G_probe"])
    Om = _dev(S.omega_matrix(150, 24, seed=8))
    beta = _beta(pp["E_probe"])
    r = 5
    P, Q, sig = _fit(lc, E, G, beta, r, Om, 0)
    P2 = torch.empty((2, 24, r), device="cuda")
    Q2 = torch.empty((2, r, 150), device="cuda")
    s2 = torch.empty((2, r), device="cuda")
    lc.loca_calib_fit(E, G, beta, r, P2, Q2, sigma=s2)
    torch.cuda.synchronize()
    P2, Q2, s2 = (t.cpu().numpy().astype(np.float64) for t in (P2, Q2, s2))
    for l in range(2):
        assert _rel(P[l] @ Q[l], P2[l] @ Q2[l]) < 1e-4
        assert _rel(sig[l], s2[l]) < 1e-5


def test_rsvd_single_probe_pair(lc):
    """Np = 1: F_hat^T = (e e^T + beta I)^-1 e g^T has rank one; the second singular value is zero
    up to the fp32 rounding of the products (1e-5 of sigma_1)."""
    pp = S.host_probe_pairs(Np=1, m=70, d=90, L=1, rank=1, seed=9)
    E, G = pp["E_probe"], pp["G_probe"]
    Om = S.omega_matrix(90, 4, seed=9)
    beta = 0.1
    P, Q, sig = _fit(lc, _dev(E), _dev(G), beta, 2, _dev(Om), 1)
    Pr, Qr, sr = O.calib_fit_rsvd(E, G, beta, 2, Om, 1)
    assert abs(sig[0, 0] - sr[0, 0]) < 1e-5 * sr[0, 0] and sig[0, 1] < 1e-5 * sr[0, 0]
    assert _rel(P[0, :, :1] @ Q[0, :1], Pr[0, :, :1] @ Qr[0, :1]) < 1e-4


def test_rsvd_reports_non_positive_definite_system(lc):
    """A NaN in the probe errors makes E^T E + beta I not positive definite in floating point:
    LOCA_ERR_NUMERIC through the status word and zero factors, not garbage."""
    rng = np.random.default_rng(4)
    E = rng.standard_normal((300, 80)).astype(np.float32)
    E[17, 5] = np.nan
    G = rng.standard_normal((2, 300, 72)).astype(np.float32)
    Om = _dev(S.omega_matrix(72, 8, seed=4))
    P = torch.full((2, 80, 4), 7.0, device="cuda")
    Q = torch.full((2, 4, 72), 7.0, device="cuda")
    sig = torch.full((2, 4), 7.0, device="cuda")
    lc.loca_device_status()
    lc.loca_calib_fit_rsvd(_dev(E), _dev(G), 0.1, 4, Om, 1, P, Q, sigma=sig)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 9
    assert torch.count_nonzero(P) == 0 and torch.count_nonzero(Q) == 0 and torch.count_nonzero(sig) == 0


def test_rsvd_full_size_sampled_block(lc):
    """Qwen2.5-7B width, the paper's d-wide error space: m = d = 3584, Np = 8192 probe tokens
    drawn on the device, r = 16 retained of a sketch of 32 with two power iterations (the
    calibration timed by the benchmark, at L = 2 here).  Block 0 against the oracle on the same
    pairs and test matrix: the planted rank-8 part of P Q to 1e-4, all 16 singular values to
    1e-5 of sigma_1."""
    Np, m, d, L, r, ell, q = 8192, 3584, 3584, 2, 16, 32, 2
    pp = S.device_probe_pairs(Np, m, d, L, rank=8, seed=1)
    E, G = pp["E_probe"], pp["G_probe"]
    Om = S.omega_matrix(d, ell, seed=1)
    beta = 1e-3 * float(torch.sum(E.double() * E.double()).item()) / m
    P, Q, sig = _fit(lc, E, G, beta, r, _dev(Om), q)
    Pr, Qr, sr = O.calib_fit_rsvd(E.cpu().numpy(), G[:1].cpu().numpy(), beta, r, Om, q)
    assert _rel(P[0, :, :8] @ Q[0, :8], Pr[0, :, :8] @ Qr[0, :8]) < 1e-4
    assert np.max(np.abs(sig[0] - sr[0])) < 1e-5 * sr[0, 0]
    assert np.allclose(Q[0] @ Q[0].T, np.eye(r), atol=1e-5)
    assert np.all(np.isfinite(P)) and np.all(np.isfinite(Q))


def test_d_wide_fit_feeds_the_label_restricted_targets(lc):
    """The paper's d-wide error space through the hot path: probe errors e = W^T eps (rows
    E_d = E_C W, W the head's C label rows, orthonormal here), fitted on the GPU with m = d and
    folded through the head (P_C = W P_d), give the label-space fit (push-through identity, same
    beta); loca_targets with the folded factors then gives the targets of the label-space fit."""
    Np, C, d, L, r = 2048, 4, 512, 2, 4
    pp = S.host_probe_pairs(Np=Np, m=C, d=d, L=L, rank=C, seed=41)
    E_C, G = pp["E_probe"], pp["G_probe"]
    rng = np.random.default_rng(41)
    W = np.linalg.qr(rng.standard_normal((d, C)))[0].T.astype(np.float32)  # C x d
    E_d = (E_C.astype(np.float64) @ W).astype(np.float32)
    beta = 0.05 * float(np.sum(E_d.astype(np.float64) ** 2)) / d
    P_d, Q_d, s_d = _fit(lc, _dev(E_d), _dev(G), beta, r, _dev(S.omega_matrix(d, 8, seed=41)), 1)
    P_fold = np.einsum("cj,ljs->lcs", W.astype(np.float64), P_d)
    P_C, Q_C, s_C, _ = O.calib_fit(E_C, G, beta, r)
    for l in range(L):
        assert _rel(P_fold[l] @ Q_d[l], P_C[l] @ Q_C[l]) < 1e-4, l
        assert np.max(np.abs(s_d[l] - s_C[l])) < 1e-5 * s_C[l, 0]
    # targets on fresh tokens: folded d-wide factors vs the GPU's label-space fit
    Pg = torch.empty((L, C, r), device="cuda")
    Qg = torch.empty((L, r, d), device="cuda")
    lc.loca_calib_fit(_dev(E_C), _dev(G), beta, r, Pg, Qg)
    E_run = _dev(rng.standard_normal((4096, C)).astype(np.float32))
    T1 = torch.empty((L, 4096, d), device="cuda")
    T2 = torch.empty((L, 4096, d), device="cuda")
    lc.loca_targets(E_run, _dev(P_fold.astype(np.float32)), _dev(Q_d.astype(np.float32)), T1)
    lc.loca_targets(E_run, Pg, Qg, T2)
    torch.cuda.synchronize()
    for l in range(L):
        assert _rel(T1[l].cpu().numpy(), T2[l].cpu().numpy().astype(np.float64)) < 1e-4, l
