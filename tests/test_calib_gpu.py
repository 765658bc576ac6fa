"""GPU parity of the one-shot calibration fit (Eq. 5; S5) against the fp64 oracle, and the
all-linear network check on the GPU path: head error -> calibration -> targets reproduce the
true backpropagated hidden-state gradients.

Tolerance: 1e-5 relative Frobenius on P Q and on each factor (the bound the statement of the
problem sets for fp32 inputs).  ``pq_bound`` derives the worst-case envelope from the arithmetic
(fp32 chunk sums of E^T E and E^T G, the conditioning of E^T E + beta I and the gap below the
retained singular values: 3.6e-5 to 4e-4 for these cases); the rounding errors are random in
sign, and the measured errors (3.5e-8 to 5.7e-8) are printed beside it.
"""

import math

import numpy as np
import pytest
import torch

from oracle import loca_oracle as O
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


def pq_bound(E, beta, F_hat, r):
    """First-order bound on the GPU fit's relative error in the rank-r map P Q.

    The inputs are exact fp32 values.  The only inexact steps before the fp64 solve are the sums
    K = E^T E and R_l = E^T G_l: fp32 products summed in fp32 over 32-token chunks (relative error
    at most u = 32 * 2^-24 per entry), chunks summed in fp64.  The solve F^T = (K + beta I)^-1 R
    multiplies a relative perturbation of K and R by at most 2 kappa(K + beta I).  The rank-r
    truncation moves by at most (1 + 2 sigma_1 / (sigma_r - sigma_{r+1})) times the perturbation
    of F (Wedin's bound for the singular subspaces, plus the values themselves).  The eigen-
    decomposition and the rest run in fp64, far below this."""
    E = np.asarray(E, dtype=np.float64)
    K = E.T @ E + beta * np.eye(E.shape[1])
    kappa = float(np.linalg.cond(K))
    s = np.linalg.svd(F_hat, compute_uv=False)
    s_next = s[r] if r < s.size else 0.0
    gap = max(s[r - 1] - s_next, 1e-300)
    return 2.0 * kappa * (32 * 2.0 ** -24) * (1.0 + 2.0 * s[0] / gap)


def _fit(lc, E, G, beta, r):
    L, Np, d = G.shape
    m = E.shape[1]
    P = torch.empty((L, m, r), device="cuda")
    Q = torch.empty((L, r, d), device="cuda")
    sig = torch.empty((L, r), device="cuda")
    lc.loca_calib_fit(_dev(E), _dev(G), beta, r, P, Q, sigma=sig)
    torch.cuda.synchronize()
    return P.cpu().numpy().astype(np.float64), Q.cpu().numpy().astype(np.float64), sig.cpu().numpy()


@pytest.mark.parametrize("Np,m,d,L,rank,r", [
    (2000, 4, 200, 2, 4, 4),
    (3000, 8, 320, 2, 8, 8),
    (4096, 16, 96, 3, 8, 8),
    (1500, 32, 130, 1, 6, 6),
    (800, 64, 72, 1, 5, 5),
])
def test_calib_parity(lc, Np, m, d, L, rank, r):
    pp = S.host_probe_pairs(Np=Np, m=m, d=d, L=L, rank=rank, seed=Np + m)
    E = pp["E_probe"]
    G = pp["G_probe"]
    beta = 1e-3 * float(np.trace(E.astype(np.float64).T @ E)) / m
    P, Q, sig = _fit(lc, E, G, beta, r)
    Pr, Qr, sr, Fh = O.calib_fit(E, G, beta, r)
    for l in range(L):
        err = _rel(P[l] @ Q[l], Pr[l] @ Qr[l])
        bound = pq_bound(E, beta, Fh[l], r)
        print(f"block {l}: P Q rel err {err:.2e}, worst-case bound of the arithmetic {bound:.2e}")
        # the fp32-input tolerance (1e-5), inside the worst-case envelope: the rounding errors of the
        # chunk sums are random in sign, so the measured error sits near 4e-8
        assert err <= min(1e-5, bound), l
        assert _rel(sig[l], sr[l]) < 1e-5
        # the factors under the sign convention
        print(f"block {l}: factor rel err Q {_rel(Q[l], Qr[l]):.2e} P {_rel(P[l], Pr[l]):.2e}")
        assert _rel(Q[l], Qr[l]) <= 1e-5 and _rel(P[l], Pr[l]) <= 1e-5
        assert np.allclose(Q[l] @ Q[l].T, np.eye(r), atol=1e-5)


def test_calib_recovers_planted_map(lc):
    """Check 3 on the GPU: exact pairs, beta -> 0: P Q recovers the planted rank-r map."""
    pp = S.host_probe_pairs(Np=4000, m=16, d=256, L=2, rank=8, noise=0.0, seed=11)
    E = pp["E_probe"]
    beta = 1e-9 * float(np.trace(E.astype(np.float64).T @ E)) / 16
    P, Q, _ = _fit(lc, E, pp["G_probe"], beta, 8)
    for l in range(2):
        assert _rel(P[l] @ Q[l], pp["M"][l]) < 1e-4


def test_linear_network_targets_equal_gradients_on_gpu(lc):
    """Check 4 on the GPU path: all-linear tokenwise network h_l = W_l h_{l-1}, z = W_u h_L.
    The true gradient is g_l = eps W_u W_L ... W_{l+1} (rows), formed here by explicit products in
    fp64.  loca_error -> loca_calib_fit(eps, g) -> loca_targets must give T_l = g_l."""
    rng = np.random.default_rng(21)
    N, d, C, Ln = 2048, 64, 4, 3
    W = [rng.standard_normal((d, d)) / math.sqrt(d) for _ in range(Ln)]
    Wu = rng.standard_normal((C, d))
    h = rng.standard_normal((N, d))
    for m in range(Ln):
        h = h @ W[m].T
    z = (h @ Wu.T).astype(np.float32)
    y = rng.integers(0, C, N).astype(np.int32)
    cols = np.arange(C, dtype=np.int32)
    E = torch.empty((N, C), device="cuda")
    lc.loca_error(_dev(z), _dev(cols, torch.int32), _dev(y, torch.int32), E)
    torch.cuda.synchronize()
    # exact gradients from the fp64 softmax of the same fp32 logits
    zz = z.astype(np.float64)
    p = np.exp(zz - zz.max(axis=1, keepdims=True))
    p /= p.sum(axis=1, keepdims=True)
    eps = p - (y[:, None] == np.arange(C)[None, :])
    grads = []
    M = Wu.copy()
    for l in range(Ln, 0, -1):  # g_l for l = Ln .. 1
        grads.append(eps @ M)
        M = M @ W[l - 1]
    grads = np.stack(grads[::-1]).astype(np.float32)  # L x N x d, g_1 .. g_L
    r = C
    P = torch.empty((Ln, C, r), device="cuda")
    Q = torch.empty((Ln, r, d), device="cuda")
    tr = float(torch.sum(E * E).item())
    # the label-set softmax rows sum to zero, so E^T E is singular; beta must sit above the
    # rounding level of its fp32-product accumulation (~1e-7 relative)
    lc.loca_calib_fit(E, _dev(grads), 1e-5 * tr / C, r, P, Q)
    T = torch.empty((Ln, N, d), device="cuda")
    lc.loca_targets(E, P, Q, T)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    for l in range(Ln):
        assert _rel(T[l].cpu().numpy(), grads[l].astype(np.float64)) < 1e-4, l


def test_calib_reports_beta_below_rounding(lc):
    """E^T E singular (columns repeated) and beta far below the fp32 rounding level: the kernel
    reports LOCA_ERR_NUMERIC through the status word and zeroes the block instead of returning
    garbage."""
    rng = np.random.default_rng(3)
    e = rng.standard_normal((512, 1)).astype(np.float32)
    E = np.concatenate([e, e, -e, 2 * e], axis=1)
    G = rng.standard_normal((1, 512, 32)).astype(np.float32)
    P = torch.full((1, 4, 2), 7.0, device="cuda")
    Q = torch.full((1, 2, 32), 7.0, device="cuda")
    lc.loca_device_status()  # clear
    lc.loca_calib_fit(_dev(E), _dev(G), 1e-30, 2, P, Q)
    torch.cuda.synchronize()
    st = lc.loca_device_status()
    if st == 0:
        # rounding happened to leave the system positive definite: outputs must then be finite
        assert torch.isfinite(P).all() and torch.isfinite(Q).all()
    else:
        assert st == 9
        assert torch.count_nonzero(P) == 0 and torch.count_nonzero(Q) == 0


@pytest.mark.parametrize("Np,m,d,L,r", [(3000, 4, 328, 3, 4), (1500, 16, 1024, 2, 16), (700, 64, 96, 1, 32),
                                         (700, 65, 96, 1, 32), (1500, 200, 256, 2, 8), (2048, 1024, 512, 2, 16)])
def test_alignment_matches_oracle(lc, Np, m, d, L, r):
    """Supplement, one-shot calibration: the in-probe cosine of each block against the oracle's.
    fp32 products summed in fp32 over 1024 tokens per thread, fp64 across: relative 1e-5.  Error
    widths above 64 (the paper's d-wide e) go through U_l = E P_l formed first."""
    rng = np.random.default_rng(Np + d)
    E = rng.standard_normal((Np, m)).astype(np.float32)
    P = rng.standard_normal((L, m, r)).astype(np.float32)
    Q = rng.standard_normal((L, r, d)).astype(np.float32)
    T = np.stack([E.astype(np.float64) @ P[l] @ Q[l] for l in range(L)])
    # gradients partly aligned with the predictions (alpha away from 0 and 1)
    G = (0.5 * T / np.sqrt(np.mean(T * T)) + rng.standard_normal((L, Np, d))).astype(np.float32)
    alpha = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_alignment(_dev(E), _dev(G), _dev(P), _dev(Q), alpha)
    torch.cuda.synchronize()
    ref = O.alignment(E, P, Q, G)
    assert np.allclose(alpha.cpu().numpy(), ref, rtol=1e-5, atol=1e-7), (alpha.cpu().numpy(), ref)


def test_alignment_of_calibrated_and_random_feedback(lc):
    """On the all-linear network the calibrated feedback reproduces the gradients (alpha ~ 1);
    random factors of the same shapes give alpha ~ 0 (the paper's contrast: -0.005 for random
    feedback, 0.3-0.5 after calibration on real models)."""
    rng = np.random.default_rng(33)
    N, d, C, Ln = 4096, 64, 4, 3
    W = [rng.standard_normal((d, d)) / math.sqrt(d) for _ in range(Ln)]
    Wu = rng.standard_normal((C, d))
    h = rng.standard_normal((N, d))
    for m_ in range(Ln):
        h = h @ W[m_].T
    z = (h @ Wu.T).astype(np.float32)
    y = rng.integers(0, C, N).astype(np.int32)
    E = torch.empty((N, C), device="cuda")
    lc.loca_error(_dev(z), _dev(np.arange(C, dtype=np.int32), torch.int32), _dev(y, torch.int32), E)
    torch.cuda.synchronize()
    E_h = E.cpu().numpy().astype(np.float64)
    grads, M = [], Wu.copy()
    for l in range(Ln, 0, -1):
        grads.append(E_h @ M)
        M = M @ W[l - 1]
    G = _dev(np.stack(grads[::-1]).astype(np.float32))
    P = torch.empty((Ln, C, C), device="cuda")
    Q = torch.empty((Ln, C, d), device="cuda")
    lc.loca_calib_fit(E, G, 1e-5 * float(torch.sum(E * E).item()) / C, C, P, Q)
    alpha = torch.empty((Ln,), dtype=torch.float64, device="cuda")
    lc.loca_alignment(E, G, P, Q, alpha)
    torch.cuda.synchronize()
    assert np.all(alpha.cpu().numpy() > 0.9999), alpha
    Pr = _dev(rng.standard_normal((Ln, C, C)).astype(np.float32))
    Qr = _dev(rng.standard_normal((Ln, C, d)).astype(np.float32))
    lc.loca_alignment(E, G, Pr, Qr, alpha)
    torch.cuda.synchronize()
    a = alpha.cpu().numpy()
    assert np.all(np.abs(a) < 0.5), a
    ref = O.alignment(E_h, Pr.cpu().numpy(), Qr.cpu().numpy(), G.cpu().numpy())
    assert np.allclose(a, ref, rtol=1e-5, atol=1e-6)
