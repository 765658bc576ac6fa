"""GPU parity of the fused-targets statistics (S3: Q_l := F_l E; S11: F e through the factors;
Eq. 9, S7) and of the closed-form ||T_l||^2 (the denominator of the step, Eq. 10), through the
C ABI, against the fp64 oracle.

``loca_gram_cross_fused`` generates each block's targets T_l = (E P_l) Q_l tile by tile on the
tensor cores and rounds them to bf16 once before they meet X, so its reference is the oracle's
cross product with the bf16-rounded targets (``t_feed="bf16"``).  The generated T carries ~2^-17
relative error before that rounding, so a few elements in a thousand round the other way than
the oracle's exact T does; that costs ~1e-4 of the cross product, inside the bf16 tolerance
(2e-3).  The Gram matrix does not involve T and must equal the default kernel's bit for bit.
"""

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


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64) if t.dtype != torch.float64 else t.cpu().numpy()


def _rel(a, b):
    a, b = np.asarray(a, dtype=np.float64), np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


def _inputs(L, N, d, C, r, seed):
    rng = np.random.default_rng(seed)
    s = rng.lognormal(0, 0.5, (L, 1, d))
    X = torch.from_numpy((rng.standard_normal((L, N, d)) * s).astype(np.float32)).to(torch.bfloat16)
    E = (rng.standard_normal((N, C)) * 0.3).astype(np.float32)
    P = rng.normal(0, 1 / np.sqrt(r), (L, C, r)).astype(np.float32)
    Q = rng.normal(0, 1 / np.sqrt(r), (L, r, d)).astype(np.float32)
    return X, E, P, Q


@pytest.mark.parametrize("L,N,d,C,r", [
    (2, 777, 328, 3, 8),
    (3, 5000, 512, 4, 16),
    (1, 64, 64, 1, 1),
    (2, 4097, 896, 16, 32),
    (2, 0, 64, 4, 4),
])
def test_targets_sq_matches_the_oracle(lc, L, N, d, C, r):
    """||E P_l Q_l||_F^2 from <P_l Q_l Q_l^T P_l^T, E^T E>: fp32 products summed in fp64, so within
    1e-6 of the oracle's sum over the formed targets."""
    _, E, P, Q = _inputs(L, N, d, C, r, seed=N + d + r)
    tsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_targets_sq(_dev(E), _dev(P), _dev(Q), tsq)
    torch.cuda.synchronize()
    _, ref = O.feedback_targets(E.astype(np.float64), P, Q)
    got = _np(tsq)
    if N == 0:
        assert np.all(got == 0.0)
    else:
        assert np.allclose(got, ref, rtol=1e-6, atol=0), (got, ref)


def _default_stats(lc, Xd, E, P, Q, alpha, zero_first, gram, cross):
    L, N, d = Xd.shape
    T = torch.empty((L, N, d), dtype=torch.bfloat16, device="cuda")
    lc.loca_targets(E, P, Q, T)
    lc.loca_gram_cross(Xd, T, alpha, gram, cross, zero_first=zero_first)


@pytest.mark.parametrize("L,d,C,r,batches", [
    (2, 328, 3, 8, (3000,)),            # d % 64 != 0 (3-D loads), ragged tiles
    (2, 512, 4, 16, (20000,)),          # two accumulation segments, 4-D loads
    (1, 640, 4, 32, (1000,)),           # r padded to 32, a partial 256-row tile
    (3, 1024, 16, 12, (5000, 3001)),    # two batches: zero_first, then accumulate; C = 16
])
def test_fused_statistics_match_the_oracle_and_the_default_kernel(lc, L, d, C, r, batches):
    f32 = dict(dtype=torch.float32, device="cuda")
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    gram_d = torch.empty((L, d, d), **f32)
    cross_d = torch.empty((L, d, d), **f32)
    g_ref = np.zeros((L, d, d))
    c_ref = np.zeros((L, d, d))
    alpha_h = np.linspace(-0.6, 0.4, L).astype(np.float32)
    alpha = _dev(alpha_h)
    Pn = Qn = None
    for b, N in enumerate(batches):
        X, E, P, Q = _inputs(L, N, d, C, r, seed=17 * N + d + b)
        if b == 0:
            Pn, Qn = P, Q
        Xd, Ed, Pd, Qd = X.to("cuda"), _dev(E), _dev(Pn), _dev(Qn)
        lc.loca_gram_cross_fused(Xd, Ed, Pd, Qd, alpha, gram, cross, zero_first=(b == 0))
        _default_stats(lc, Xd, Ed, Pd, Qd, alpha, b == 0, gram_d, cross_d)
        torch.cuda.synchronize()
        Xn = X.float().numpy().astype(np.float64)
        T, _ = O.feedback_targets(E.astype(np.float64), Pn, Qn)
        for l in range(L):
            g_ref[l] += Xn[l].T @ Xn[l]
            c_ref[l] += float(alpha_h[l]) * (O.round_to_bf16(T[l]).T @ Xn[l])
    assert lc.loca_device_status() == 0
    rg, rc = _rel(_np(gram), g_ref), _rel(_np(cross), c_ref)
    rcd = _rel(_np(cross), _np(cross_d))
    print(f"fused: rel err gram {rg:.2e} cross {rc:.2e}; cross vs default kernel {rcd:.2e}")
    assert torch.equal(gram, gram_d)  # the Gram tiles are the same products in the same order
    gg = _np(gram)
    assert np.array_equal(gg, np.transpose(gg, (0, 2, 1)))
    assert rg <= 1e-4 and rc <= 2e-3 and rcd <= 2e-3


def test_fused_statistics_are_deterministic(lc):
    L, N, d, C, r = 2, 9000, 768, 4, 16
    X, E, P, Q = _inputs(L, N, d, C, r, seed=4)
    args = (X.to("cuda"), _dev(E), _dev(P), _dev(Q), _dev(np.array([0.5, -1.0], dtype=np.float32)))
    outs = []
    for _ in range(2):
        gram = torch.empty((L, d, d), device="cuda")
        cross = torch.empty((L, d, d), device="cuda")
        lc.loca_gram_cross_fused(*args, gram, cross, zero_first=True)
        outs.append((gram.clone(), cross.clone()))
    torch.cuda.synchronize()
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_fused_chain_at_the_qwen7b_shape(lc):
    """The 7B workload (L = 28, N = 131072, d = 3584, r = k = 16) through the fused chain:
    error -> ||T||^2 in closed form -> fused statistics at alpha = 1 -> step from the Gram trace ->
    solve with alpha applied; against the default chain on the same inputs (Gram identical, cross
    product and adapters within the bf16 tolerance) and against the oracle on the last block."""
    w = S.WORKLOADS["qwen2.5-7b"]
    inp = S.device_inputs(w, seed=0, device="cuda")
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, k = w.L, w.N, w.d, w.C, w.k
    nl = len(w.lambda_rel)
    f32 = dict(dtype=torch.float32, device="cuda")
    E = torch.empty((N, C), **f32)
    lc.loca_error(z, cols, y, E)
    ones = torch.ones((L,), **f32)
    out = {}
    for mode in ("fused", "default"):
        gram = torch.empty((L, d, d), **f32)
        cross = torch.empty((L, d, d), **f32)
        tsq = torch.empty((L,), dtype=torch.float64, device="cuda")
        xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
        alpha = torch.empty((L,), **f32)
        B = torch.empty((nl, L, d, k), **f32)
        info = torch.empty((nl, L), dtype=torch.int32, device="cuda")
        if mode == "fused":
            lc.loca_targets_sq(E, P, Q, tsq)
            lc.loca_gram_cross_fused(X, E, P, Q, ones, gram, cross, zero_first=True)
        else:
            T = torch.empty((L, N, d), dtype=torch.bfloat16, device="cuda")
            lc.loca_targets(E, P, Q, T, tsq=tsq)
            lc.loca_gram_cross(X, T, ones, gram, cross, zero_first=True)
            del T
        lc.loca_step_from_gram(gram, tsq, w.eta, xsq, alpha)
        lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, cross_scale=alpha)
        torch.cuda.synchronize()
        assert lc.loca_device_status() == 0 and int(info.abs().sum()) == 0
        out[mode] = dict(gram=gram, cross=cross, tsq=tsq, alpha=alpha, B=B)
    fu, de = out["fused"], out["default"]
    assert torch.equal(fu["gram"], de["gram"])
    assert np.allclose(_np(fu["tsq"]), _np(de["tsq"]), rtol=1e-5, atol=0)
    for l in (0, L - 1):
        rc = _rel(_np(fu["cross"][l]), _np(de["cross"][l]))
        rb = max(_rel(_np(fu["B"][j, l]), _np(de["B"][j, l])) for j in range(nl))
        print(f"block {l}: fused vs default, cross {rc:.2e}, B {rb:.2e}")
        assert rc <= 2e-3 and rb <= 2e-3
    h = inp["host"]
    l = L - 1
    E_ref, _ = O.head_error(_np(z), h["label_cols"], h["y"])
    X_h = _np(X[l])[None]
    ref = O.loca_pass(_np(z), h["label_cols"], h["y"], X_h, h["P"][l:l + 1], h["Q"][l:l + 1], h["A"][l:l + 1],
                      w.eta, w.lambda_rel, t_feed="bf16")
    rc = _rel(_np(fu["cross"][l]) * float(fu["alpha"][l]), ref["cross"][0])
    rb = max(_rel(_np(fu["B"][j, l]), ref["B"][j, 0]) for j in range(nl))
    assert abs(float(fu["tsq"][l]) - ref["tsq"][0]) <= 1e-6 * ref["tsq"][0]
    print(f"block {l}: fused vs oracle, cross {rc:.2e}, B {rb:.2e}")
    assert rc <= 2e-3 and rb <= 2e-3
    del out, fu, de, inp, X
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
