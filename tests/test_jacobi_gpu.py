"""The Jacobi outer loop (S13 steps 2-5; S8) run through the C ABI on a small all-linear network.

Network (tokenwise, no attention): h_l = W_l h_{l-1} + B_l A_l^T h_{l-1}, z = W_u h_L, with
frozen W_l, W_u and fixed A_l; labels come from a teacher whose perturbation B*_l A_l^T lies in
the adapters' span.  The feedback factors are calibrated once at the frozen model from the true
gradients (S5).  Each outer iteration: forward (numpy, fp64; the frozen backbone is not part of
the library) -> loca_error -> loca_targets -> loca_accumulate -> loca_ridge_solve with
B_prev = the current adapters.  Checked at every iteration:

* B from the GPU equals the oracle's chain on the same inputs (relative 1e-4);
* every block's local objective J_l(B) = ||B P - R||^2 + lambda ||B||^2 does not increase, and
  the decrease equals tr(D (G + lambda I) D^T) with D = B_new - B_prev (the gap identity,
  Theorem S6), from the G_l, C_l the solve reports;

and over the run the training cross-entropy goes down (the paper claims no global
monotonicity; this checks the method learns where it can, not a guarantee).
"""

import math

import numpy as np
import pytest
import torch

from oracle import loca_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    from paper_2608_03020_gb300 import loca

    loca.lib()
    return loca


def _dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


def _forward(h0, W, A, B, Wu):
    X, h = [], h0
    for l in range(len(W)):
        X.append(h)
        h = h @ W[l].T + (h @ A[l]) @ B[l].T
    return np.stack(X), h @ Wu.T


def test_jacobi_outer_loop_all_linear(lc):
    rng = np.random.default_rng(11)
    L, d, N, C, k = 3, 64, 4096, 4, 8
    r = C
    eta, lam_rel = 0.05, [1e-3]
    W = [np.linalg.qr(rng.standard_normal((d, d)))[0] for _ in range(L)]
    Wu = rng.standard_normal((C, d))
    A = np.stack([np.linalg.qr(rng.standard_normal((d, k)))[0] for _ in range(L)])
    h0 = rng.standard_normal((N, d))
    B_teacher = [0.6 * rng.standard_normal((d, k)) / math.sqrt(k) for _ in range(L)]
    _, z_t = _forward(h0, W, A, B_teacher, Wu)
    y = np.argmax(z_t, axis=1).astype(np.int32)
    cols = np.arange(C, dtype=np.int32)

    # calibration at the frozen model from the true gradients g_l = eps W_u W_L ... W_{l+1}
    B = np.zeros((L, d, k))
    X, z = _forward(h0, W, A, B, Wu)
    z32 = z.astype(np.float32)
    E = torch.empty((N, C), device="cuda")
    lc.loca_error(_dev(z32), _dev(cols, torch.int32), _dev(y, torch.int32), E)
    torch.cuda.synchronize()
    E_h = E.cpu().numpy().astype(np.float64)
    grads, M = [], Wu.copy()
    for l in range(L, 0, -1):
        grads.append(E_h @ M)
        M = M @ W[l - 1]
    grads = np.stack(grads[::-1]).astype(np.float32)
    P = torch.empty((L, C, r), device="cuda")
    Q = torch.empty((L, r, d), device="cuda")
    tr = float(torch.sum(E * E).item())
    lc.loca_calib_fit(E, _dev(grads), 1e-5 * tr / C, r, P, Q)
    torch.cuda.synchronize()
    P_h, Q_h = P.cpu().numpy(), Q.cpu().numpy()

    f32 = dict(device="cuda", dtype=torch.float32)
    T = torch.empty((L, N, d), **f32)
    tsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    Bn = torch.empty((1, L, d, k), **f32)
    info = torch.empty((1, L), dtype=torch.int32, device="cuda")
    G_out = torch.empty((L, k, k), **f32)
    C_out = torch.empty((L, d, k), **f32)
    ce = torch.empty((N,), **f32)
    losses = []
    for t in range(6):
        X, z = _forward(h0, W, A, B, Wu)
        X32, z32 = X.astype(np.float32), z.astype(np.float32)
        B32 = B.astype(np.float32)
        lc.loca_error(_dev(z32), _dev(cols, torch.int32), _dev(y, torch.int32), E, ce=ce)
        lc.loca_targets(E, P, Q, T, tsq=tsq)
        lc.loca_accumulate(_dev(X32), T, tsq, eta, gram, cross, xsq, zero_first=True)
        lc.loca_ridge_solve(gram, cross, _dev(A.astype(np.float32)), lam_rel, Bn, info, xsq_total=xsq,
                            B_prev=_dev(B32), G_out=G_out, C_out=C_out)
        torch.cuda.synchronize()
        assert lc.loca_device_status() == 0 and int(info.abs().sum()) == 0
        losses.append(float(ce.mean().item()))
        ref = O.loca_pass(z32, cols, y, X32, P_h, Q_h, A.astype(np.float32), eta, lam_rel, B_prev=B32)
        B_new = Bn[0].cpu().numpy().astype(np.float64)
        rel = np.linalg.norm(B_new - ref["B"][0]) / np.linalg.norm(ref["B"][0])
        assert rel < 1e-4, (t, rel)
        # local objective of each block (up to its constant): tr(B (G + lam I) B^T) - 2 tr(C B^T)
        G = G_out.cpu().numpy().astype(np.float64)
        Cm = C_out.cpu().numpy().astype(np.float64)
        lam = lam_rel[0] * xsq.cpu().numpy() / d
        for l in range(L):
            H = G[l] + lam[l] * np.eye(k)

            def J(Bx):
                return float(np.trace(Bx @ H @ Bx.T) - 2.0 * np.trace(Cm[l] @ Bx.T))

            D = B_new[l] - B32[l].astype(np.float64)
            drop = J(B32[l].astype(np.float64)) - J(B_new[l])
            gap = float(np.trace(D @ H @ D.T))
            assert drop >= -1e-6 * max(abs(J(B_new[l])), 1.0), (t, l, drop)
            assert abs(drop - gap) <= 1e-3 * gap + 1e-9, (t, l, drop, gap)
        B = B_new
    print("training CE per outer iteration:", " ".join(f"{v:.4f}" for v in losses))
    assert losses[-1] < 0.9 * losses[0]
