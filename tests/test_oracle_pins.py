"""Pins of the fp64 oracle against facts fixed by the paper and by mathematics.

Each test checks the oracle against something other than itself: hand-derived closed
forms (``tests/golden/closed_forms.json``), brute-force loops, finite differences of the
paper's losses, textbook library routines, and identities the paper proves.  A dropped
term, a wrong sign or index, or a transposed operand in the oracle fails at least one.
"""

import json
import math
import os

import numpy as np
import pytest
from scipy.special import logsumexp

from oracle import loca_oracle as O
from synth import inputs as S

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "closed_forms.json")))


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


# ---------------------------------------------------------------- bf16 storage rounding

def test_bf16_rounding_matches_torch_and_ties_to_even():
    import torch

    rng = np.random.default_rng(1)
    x = (rng.standard_normal(20000) * np.exp(rng.uniform(-20, 20, 20000))).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(O.round_to_bf16(x.astype(np.float64)), ref)
    # ties: 1 + 2^-8 lies halfway between 1 and 1 + 2^-7 -> even (1); 1 + 3*2^-8 -> 1 + 2^-6
    assert O.round_to_bf16(1.0 + 2.0 ** -8) == 1.0
    assert O.round_to_bf16(1.0 + 3 * 2.0 ** -8) == 1.0 + 2.0 ** -6
    assert O.round_to_bf16(-(1.0 + 3 * 2.0 ** -8)) == -(1.0 + 2.0 ** -6)
    assert O.round_to_bf16(0.0) == 0.0


# ---------------------------------------------------------------- O1 head error

@pytest.mark.parametrize("case", range(len(GOLDEN["head_error"])))
def test_head_error_closed_forms(case):
    g = GOLDEN["head_error"][case]
    E, ce = O.head_error(np.array(g["z"]), g["label_cols"], np.array(g["y"]),
                         w=None if g["w"] is None else np.array(g["w"]), normaliser=g["normaliser"])
    assert np.allclose(E, g["E"], atol=1e-14)
    assert np.allclose(ce, g["ce"], atol=1e-14)


def _ce_direct(z, cols, y, w, normaliser):
    """Per-token weighted cross-entropy written from the loss of S3 (scipy logsumexp)."""
    out = np.zeros(z.shape[0])
    for n in range(z.shape[0]):
        if y[n] < 0:
            continue
        row = z[n] if normaliser == 0 else z[n, cols]
        out[n] = w[n] * (logsumexp(row) - z[n, cols[y[n]]])
    return out


@pytest.mark.parametrize("normaliser", [0, 1])
def test_head_error_is_derivative_of_cross_entropy(normaliser):
    """Lemma S3: E[n, c] = d(w_n CE_n)/d z_{n, label_cols[c]}, by central differences."""
    rng = np.random.default_rng(2)
    N, V = 6, 9
    cols = np.array([1, 4, 6, 8])
    z = rng.standard_normal((N, V)) * 2.0
    y = rng.integers(0, cols.size, N)
    y[3] = -1
    w = rng.uniform(0.5, 2.0, N)
    E, ce = O.head_error(z, cols, y, w=w, normaliser=normaliser)
    assert np.allclose(ce, _ce_direct(z, cols, y, w, normaliser), atol=1e-13)
    h = 1e-6
    for n in range(N):
        for c, col in enumerate(cols):
            zp, zm = z.copy(), z.copy()
            zp[n, col] += h
            zm[n, col] -= h
            fd = (_ce_direct(zp, cols, y, w, normaliser)[n] - _ce_direct(zm, cols, y, w, normaliser)[n]) / (2 * h)
            assert abs(fd - E[n, c]) < 1e-8
    assert np.all(E[3] == 0.0) and ce[3] == 0.0


def test_head_error_row_sums_and_bounds():
    """With the label normaliser the softmax and the one-hot both sum to one over the
    labels, so each row of E sums to zero; E[n, y_n] lies in (-1, 0]."""
    rng = np.random.default_rng(3)
    z = rng.standard_normal((50, 5)) * 3
    y = rng.integers(0, 3, 50)
    E, _ = O.head_error(z, [0, 2, 4], y, normaliser=1)
    assert np.allclose(E.sum(axis=1), 0.0, atol=1e-14)
    Ey = E[np.arange(50), y]
    assert np.all(Ey <= 0) and np.all(Ey > -1)
    # the full-row normaliser gives a sum in (-1, 0] (non-label columns hold the rest)
    E0, _ = O.head_error(z, [0, 2, 4], y, normaliser=0)
    assert np.all(E0.sum(axis=1) <= 1e-15) and np.all(E0.sum(axis=1) > -1)


def test_head_error_brute_force_all_labelings():
    """Enumerate every labelling y in {0,1}^3 of a 3-token, 2-class case: the gradient of
    the summed loss (central differences) equals the stacked error."""
    rng = np.random.default_rng(4)
    z = rng.standard_normal((3, 2))
    cols = np.array([0, 1])
    w = np.ones(3)
    h = 1e-6
    for lab in range(8):
        y = np.array([(lab >> b) & 1 for b in range(3)])
        E, _ = O.head_error(z, cols, y)
        for n in range(3):
            for c in range(2):
                zp, zm = z.copy(), z.copy()
                zp[n, c] += h
                zm[n, c] -= h
                fd = (_ce_direct(zp, cols, y, w, 0).sum() - _ce_direct(zm, cols, y, w, 0).sum()) / (2 * h)
                assert abs(fd - E[n, c]) < 1e-8


def test_head_error_c2_is_sigmoid():
    """Two classes, label normaliser: E[n,0] = sigmoid(z0 - z1) - 1[y=0]."""
    rng = np.random.default_rng(5)
    z = rng.standard_normal((40, 2)) * 4
    y = rng.integers(0, 2, 40)
    E, _ = O.head_error(z, [0, 1], y, normaliser=1)
    sig = 1.0 / (1.0 + np.exp(-(z[:, 0] - z[:, 1])))
    assert np.allclose(E[:, 0], sig - (y == 0), atol=1e-14)


def test_head_error_large_logits_stable():
    z = np.array([[1000.0, 1001.0, -1000.0]])
    E, ce = O.head_error(z, [0, 1, 2], np.array([1]))
    p = np.array([1 / (1 + math.e), math.e / (1 + math.e), 0.0])
    assert np.allclose(E[0], p - np.array([0, 1, 0]), atol=1e-14)
    assert np.isfinite(ce).all()


# ---------------------------------------------------------------- O2 targets

def test_targets_brute_force_loops():
    rng = np.random.default_rng(6)
    L, N, C, r, d = 2, 4, 3, 2, 5
    E = rng.standard_normal((N, C))
    P = rng.standard_normal((L, C, r))
    Q = rng.standard_normal((L, r, d))
    T, tsq = O.feedback_targets(E, P, Q)
    for l in range(L):
        acc_sq = 0.0
        for n in range(N):
            for j in range(d):
                v = 0.0
                for c in range(C):
                    for s in range(r):
                        v += E[n, c] * P[l, c, s] * Q[l, s, j]
                assert abs(T[l, n, j] - v) < 1e-12
                acc_sq += v * v
        assert abs(tsq[l] - acc_sq) < 1e-10


# ---------------------------------------------------------------- O3 statistics

def test_stats_closed_form():
    g = GOLDEN["stats"][0]
    X = np.array(g["X"])[None]
    T = np.array(g["T"])[None]
    assert abs(O.scaled_step(g["eta"], X[0], T[0]) - g["eta_bar"]) < 1e-15
    gram, cross, xsq = O.accumulate_stats([X], [T], g["eta"])
    assert np.allclose(gram[0], g["gram"]) and np.allclose(cross[0], g["cross"]) and abs(xsq[0] - g["xsq"]) < 1e-14
    r = GOLDEN["rms"][0]
    assert abs(O.rms(np.array(r["X"])) - r["rms"]) < 1e-14


def test_stats_brute_force_loops():
    rng = np.random.default_rng(7)
    N, d, eta = 6, 3, 0.03
    X = rng.standard_normal((1, N, d))
    T = rng.standard_normal((1, N, d))
    gram, cross, xsq = O.accumulate_stats([X], [T], eta)
    sx = sum(X[0, n, j] ** 2 for n in range(N) for j in range(d))
    st = sum(T[0, n, j] ** 2 for n in range(N) for j in range(d))
    step = eta * math.sqrt(sx / (N * d)) / math.sqrt(st / (N * d))
    for i in range(d):
        for j in range(d):
            gij = sum(X[0, n, i] * X[0, n, j] for n in range(N))
            cij = -step * sum(T[0, n, i] * X[0, n, j] for n in range(N))
            assert abs(gram[0, i, j] - gij) < 1e-12
            assert abs(cross[0, i, j] - cij) < 1e-12
    assert abs(xsq[0] - sx) < 1e-12


def test_stats_bf16_feed_rounds_only_the_cross_operand():
    rng = np.random.default_rng(8)
    X = rng.standard_normal((1, 20, 4))
    T = rng.standard_normal((1, 20, 4)) * 0.37
    _, c_exact, _ = O.accumulate_stats([X], [T], 0.01)
    _, c_bf, _ = O.accumulate_stats([X], [T], 0.01, t_feed="bf16")
    step = O.scaled_step(0.01, X[0], T[0])  # unrounded T sets the step
    Tr = O.round_to_bf16(T[0])
    ref = np.zeros((4, 4))
    for n in range(20):
        ref += -step * np.outer(Tr[n], X[0, n])
    assert np.allclose(c_bf[0], ref, rtol=0, atol=1e-14)
    assert not np.allclose(c_bf, c_exact, rtol=0, atol=1e-12)


def test_scale_invariance_of_target_prop_s8():
    """Prop. S8: Q -> aQ (a > 0) leaves the displacement -eta_bar Q, hence Cross, unchanged;
    and RMS(-eta_bar Q) = eta RMS(H)."""
    rng = np.random.default_rng(9)
    X = rng.standard_normal((2, 30, 5)) * 3
    T = rng.standard_normal((2, 30, 5))
    _, c1, _ = O.accumulate_stats([X], [T], 0.03)
    _, c2, _ = O.accumulate_stats([X], [T * 7.25], 0.03)
    assert _rel(c2, c1) < 1e-14
    for l in range(2):
        step = O.scaled_step(0.03, X[l], T[l])
        assert abs(O.rms(-step * T[l]) - 0.03 * O.rms(X[l])) < 1e-14


def test_zero_targets_give_zero_step():
    X = np.ones((1, 4, 3))
    T = np.zeros((1, 4, 3))
    assert O.scaled_step(0.01, X[0], T[0]) == 0.0
    _, cross, _ = O.accumulate_stats([X], [T], 0.01)
    assert np.all(cross == 0.0)


def _per_token_stats(X, T_batches, batch_of, eta, A, B_prev):
    """Paper-side definitions per token: p = A^T x, q = the target row, rho = B p - s q with
    s the step of the token's mini-batch (Eqs. 6, 9, 10; S7, S8)."""
    L, N, d = X.shape
    k = A.shape[2]
    Tall = np.concatenate(T_batches, axis=1)
    G = np.zeros((L, k, k))
    C = np.zeros((L, d, k))
    for l in range(L):
        steps = []
        for m, Tm in enumerate(T_batches):
            idx = np.where(batch_of == m)[0]
            xs = X[l, idx]
            ts = Tm[l]
            sx = math.sqrt(np.sum(xs ** 2) / xs.size)
            st = math.sqrt(np.sum(ts ** 2) / ts.size)
            steps.append(0.0 if st == 0 else eta * sx / st)
        for n in range(N):
            p = A[l].T @ X[l, n]
            q = Tall[l, n]
            rho = (B_prev[l] @ p if B_prev is not None else 0.0) - steps[batch_of[n]] * q
            G[l] += np.outer(p, p)
            C[l] += np.outer(rho, p)
    return G, C


def test_streaming_and_projection_match_per_token_definitions():
    """Streaming additivity (S7) with one step per mini-batch (S8), and projection onto the
    adapter features (Eq. 9): the d x d route equals the per-token k-space sums."""
    rng = np.random.default_rng(10)
    L, N, d, k, C, r = 2, 21, 6, 3, 3, 2
    X = rng.standard_normal((L, N, d)) * rng.lognormal(0, 0.5, (L, 1, d))
    E = rng.standard_normal((N, C))
    P = rng.standard_normal((L, C, r))
    Q = rng.standard_normal((L, r, d))
    A = np.stack([np.linalg.qr(rng.standard_normal((d, k)))[0] for _ in range(L)])
    Bp = rng.standard_normal((L, d, k)) * 0.1
    bounds = [0, 8, 15, 21]
    batch_of = np.zeros(N, dtype=int)
    Xb, Tb = [], []
    for m in range(3):
        s = slice(bounds[m], bounds[m + 1])
        batch_of[s] = m
        Tm, _ = O.feedback_targets(E[s], P, Q)
        Xb.append(X[:, s])
        Tb.append(Tm)
    gram, cross, xsq = O.accumulate_stats(Xb, Tb, 0.01)
    G, Cst = O.project_stats(gram, cross, A, B_prev=Bp)
    G_ref, C_ref = _per_token_stats(X, Tb, batch_of, 0.01, A, Bp)
    assert _rel(G, G_ref) < 1e-13 and _rel(Cst, C_ref) < 1e-13
    assert np.allclose(xsq, [np.trace(gram[l]) for l in range(L)], rtol=1e-14)
    # one-shot Gram equals the streamed Gram (additivity)
    g1, _, _ = O.accumulate_stats([X], [np.concatenate(Tb, axis=1)], 0.01)
    assert _rel(g1, gram) < 1e-14
    # the paper's own k x k / d x k statistics, accumulated without a d x d matrix
    Gk, Ck, xk = O.kspace_stats(Xb, Tb, A, 0.01, B_prev=Bp)
    assert _rel(Gk, G_ref) < 1e-13 and _rel(Ck, C_ref) < 1e-13
    assert np.allclose(xk, xsq, rtol=1e-14)


def test_kspace_stats_brute_force_and_special_cases():
    """kspace_stats against per-token loops without B_prev (rho = -eta_bar q), the zero-target
    case (no step, C = B_prev G), Prop. S8 (T -> aT leaves C unchanged) and a feature map that
    is the identity (G is then the Gram of X)."""
    rng = np.random.default_rng(12)
    L, N, d, k, C, r = 2, 17, 5, 2, 3, 2
    X = rng.standard_normal((L, N, d))
    E = rng.standard_normal((N, C))
    P = rng.standard_normal((L, C, r))
    Q = rng.standard_normal((L, r, d))
    A = rng.standard_normal((L, d, k))
    T, _ = O.feedback_targets(E, P, Q)
    G, Cs, _ = O.kspace_stats([X], [T], A, 0.03)
    G_ref, C_ref = _per_token_stats(X, [T], np.zeros(N, dtype=int), 0.03, A, None)
    assert _rel(G, G_ref) < 1e-13 and _rel(Cs, C_ref) < 1e-13
    Bp = rng.standard_normal((L, d, k))
    G0, C0, _ = O.kspace_stats([X], [np.zeros_like(T)], A, 0.03, B_prev=Bp)
    assert np.allclose(C0, np.einsum("ldk,lkj->ldj", Bp, G0), rtol=1e-13, atol=1e-12)
    _, C2, _ = O.kspace_stats([X], [4.0 * T], A, 0.03)
    assert _rel(C2, Cs) < 1e-13
    eye = np.stack([np.eye(d)] * L)
    Gi, _, _ = O.kspace_stats([X], [T], eye, 0.03)
    assert np.allclose(Gi, np.einsum("lnd,lne->lde", X, X), rtol=1e-13, atol=1e-12)


# ---------------------------------------------------------------- O5 solve

def test_cholesky_closed_form_and_not_pd():
    g = GOLDEN["cholesky"][0]
    Lo, info = O.cholesky(np.array(g["M"]))
    assert info == 0 and np.allclose(Lo, g["L"], atol=1e-15)
    _, info = O.cholesky(-np.eye(3))
    assert info == 1
    _, info = O.cholesky(np.array([[1.0, 2.0], [2.0, 1.0]]))
    assert info == 2


@pytest.mark.parametrize("case", range(len(GOLDEN["ridge"])))
def test_ridge_closed_forms(case):
    g = GOLDEN["ridge"][case]
    B, info = O.ridge_solve(np.array(g["G"])[None], np.array(g["C"])[None], np.array([[g["lambda"]]]))
    assert info[0, 0] == 0 and np.allclose(B[0, 0], g["B"], atol=1e-14)


def _ridge_problem(seed=11, N=40, d=7, k=4):
    rng = np.random.default_rng(seed)
    Pm = rng.standard_normal((N, k)) * np.array([3.0, 1.0, 0.5, 0.2])[:k]
    R = rng.standard_normal((N, d))
    G = (Pm.T @ Pm)[None]
    C = (R.T @ Pm)[None]
    return Pm, R, G, C


def test_ridge_normal_equations_and_textbook_solve():
    Pm, R, G, C = _ridge_problem()
    lam = np.array([[0.3], [5.0]])
    B, info = O.ridge_solve(G, C, lam)
    k = G.shape[1]
    for j in range(2):
        lhs = B[j, 0] @ (G[0] + lam[j, 0] * np.eye(k))
        assert _rel(lhs, C[0]) < 1e-13  # normal equations (check 1)
        ref = np.linalg.solve(G[0] + lam[j, 0] * np.eye(k), C[0].T).T
        assert _rel(B[j, 0], ref) < 1e-13
    assert np.all(info == 0)


def test_ridge_limits_lambda_to_infinity_and_zero():
    """Check 2: lambda -> inf gives B -> 0 like C / lambda; lambda -> 0 gives the least-squares
    fit of the per-token problem min_B sum ||B p_n - rho_n||^2 (numpy.linalg.lstsq)."""
    Pm, R, G, C = _ridge_problem()
    big = 1e9 * np.trace(G[0])
    B, _ = O.ridge_solve(G, C, np.array([[big]]))
    assert _rel(big * B[0, 0], C[0]) < 1e-8
    assert np.linalg.norm(B) < 1e-8 * np.linalg.norm(C) / np.trace(G[0]) * 10
    B0, _ = O.ridge_solve(G, C, np.array([[1e-13 * np.trace(G[0])]]))
    Bls = np.linalg.lstsq(Pm, R, rcond=None)[0].T
    assert _rel(B0[0, 0], Bls) < 1e-9


def test_ridge_gap_identity():
    """Theorem S6: Phi(B) - Phi(B*) = tr((B - B*)(G + lambda I)(B - B*)^T), Phi per token."""
    Pm, R, G, C = _ridge_problem()
    lam = 0.7
    Bs, _ = O.ridge_solve(G, C, np.array([[lam]]))
    Bs = Bs[0, 0]

    def phi(B):
        return sum(np.sum((B @ Pm[n] - R[n]) ** 2) for n in range(Pm.shape[0])) + lam * np.sum(B * B)

    rng = np.random.default_rng(12)
    for _ in range(5):
        B = Bs + rng.standard_normal(Bs.shape) * 0.3
        D = B - Bs
        gap = np.trace(D @ (G[0] + lam * np.eye(G.shape[1])) @ D.T)
        assert abs((phi(B) - phi(Bs)) - gap) < 1e-9 * max(1.0, gap)
        assert phi(B) > phi(Bs)


def test_lambdas_relative_to_trace():
    lam = O.ridge_lambdas([1e-4, 1e-2], np.array([10.0, 30.0]), 5)
    assert np.allclose(lam, [[2e-4, 6e-4], [2e-2, 6e-2]])
    lam_abs = O.ridge_lambdas([0.5], None, 5)
    assert lam_abs.shape == (1, 1) and lam_abs[0, 0] == 0.5


def test_pass_scale_invariance_with_relative_lambda():
    """X -> aX with B_prev = 0 and lambda proportional to tr(Gram)/d leaves B* unchanged:
    Gram, lambda and Cross all scale by a^2 (S8 step, Eq. 8)."""
    w = S.scaled(S.WORKLOADS["tiny"], N=96, d=16, r=3, k=3)
    f = S.host_inputs(w)
    a = 3.5
    o1 = O.loca_pass(f["z"], f["label_cols"], f["y"], f["X"], f["P"], f["Q"], f["A"], 0.01, [1e-3, 1e-1])
    o2 = O.loca_pass(f["z"], f["label_cols"], f["y"], a * f["X"].astype(np.float64), f["P"], f["Q"], f["A"], 0.01,
                     [1e-3, 1e-1])
    assert _rel(o2["B"], o1["B"]) < 1e-12
    assert _rel(o2["gram"], a * a * o1["gram"]) < 1e-13


def test_pass_end_to_end_first_order_condition():
    """The full pass's B* makes the per-token ridge objective stationary: the per-token
    objective is assembled from finite-difference head errors (Lemma S3), explicit token
    loops for q, p and rho (Eqs. 6, 9), the step of Eq. 10 and lambda = c tr(Gram)/d."""
    w = S.scaled(S.WORKLOADS["tiny"], L=2, N=24, d=6, r=2, k=2, C=3, V=3)
    f = S.host_inputs(w)
    X = f["X"].astype(np.float64)
    Bp = S.host_B_prev(w) * 10
    out = O.loca_pass(f["z"], f["label_cols"], f["y"], X, f["P"], f["Q"], f["A"], 0.02, [0.05], B_prev=Bp)
    z = f["z"].astype(np.float64)
    cols = f["label_cols"]
    y = f["y"]
    N, d = X.shape[1], X.shape[2]
    h = 1e-6
    e = np.zeros((N, w.C))
    for n in range(N):
        for c in range(w.C):
            zp, zm = z.copy(), z.copy()
            zp[n, cols[c]] += h
            zm[n, cols[c]] -= h
            e[n, c] = (_ce_direct(zp, cols, y, np.ones(N), 0)[n] - _ce_direct(zm, cols, y, np.ones(N), 0)[n]) / (2 * h)
    for l in range(w.L):
        q = np.array([[sum(e[n, c] * f["P"][l, c, s] * f["Q"][l, s, j] for c in range(w.C) for s in range(w.r))
                       for j in range(d)] for n in range(N)])
        step = 0.02 * math.sqrt(np.mean(X[l] ** 2)) / math.sqrt(np.mean(q ** 2))
        p = X[l] @ f["A"][l].astype(np.float64)
        rho = p @ Bp[l].astype(np.float64).T - step * q
        lam = 0.05 * np.sum(X[l] ** 2) / d
        B = out["B"][0, l]
        grad = 2 * (B @ p.T - rho.T) @ p + 2 * lam * B  # d Phi / dB of the per-token objective
        assert np.linalg.norm(grad) < 1e-6 * (np.linalg.norm(rho.T @ p) + 1.0)


# ---------------------------------------------------------------- O6 calibration

def test_calib_primal_equals_dual():
    pp = S.host_probe_pairs(Np=30, m=6, d=9, L=2, rank=3, seed=3)
    _, _, _, Fh = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.5, 4)
    Fd = O.calib_fit_dual(pp["E_probe"], pp["G_probe"], 0.5)
    assert _rel(Fh, Fd) < 1e-12


def test_calib_recovers_planted_rank_map():
    """Check 3: with exact pairs (no noise) and beta -> 0 the rank-r truncation of the fit
    equals the planted rank-r map."""
    pp = S.host_probe_pairs(Np=80, m=8, d=12, L=2, rank=4, noise=0.0, seed=4)
    E = pp["E_probe"].astype(np.float64)
    beta = 1e-12 * np.trace(E.T @ E) / 8
    P, Q, sig, _ = O.calib_fit(E, E @ pp["M"][0][None].repeat(1, 0), beta, 4)
    assert _rel(P[0] @ Q[0], pp["M"][0]) < 1e-8
    # orthonormal rows of Q, sign convention
    assert np.allclose(Q[0] @ Q[0].T, np.eye(4), atol=1e-12)
    for i in range(4):
        assert Q[0, i, np.argmax(np.abs(Q[0, i]))] > 0
    assert np.all(np.diff(sig[0]) <= 0)


def test_calib_rank_truncation_lemma():
    """Lemma S5: ||F_hat - F||_F^2 = sum_{j>r} sigma_j^2 and ||(F_hat - F) e|| <= sigma_{r+1} ||e||."""
    pp = S.host_probe_pairs(Np=50, m=7, d=10, L=1, rank=7, seed=5)
    _, _, sig_full, Fh = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.1, 7)
    r = 3
    P, Q, _, _ = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.1, r)
    Fr = P[0] @ Q[0]
    assert abs(np.sum((Fh[0] - Fr) ** 2) - np.sum(sig_full[0, r:] ** 2)) < 1e-10 * np.sum(sig_full[0] ** 2)
    rng = np.random.default_rng(6)
    for _ in range(20):
        e = rng.standard_normal(7)
        assert np.linalg.norm(e @ (Fh[0] - Fr)) <= sig_full[0, r] * np.linalg.norm(e) * (1 + 1e-12)


def test_calib_is_stationary_point_of_ridge_objective():
    """Eq. 5: the fit minimises ||F E - G||^2 + beta ||F||^2; directional derivatives at
    F_hat vanish (central differences of the objective)."""
    pp = S.host_probe_pairs(Np=25, m=4, d=6, L=1, rank=2, seed=7)
    E = pp["E_probe"].astype(np.float64)
    G = pp["G_probe"][0].astype(np.float64)
    beta = 0.3
    _, _, _, Fh = O.calib_fit(E, pp["G_probe"], beta, 4)
    Ft = Fh[0]

    def J(Ft_):
        return np.sum((E @ Ft_ - G) ** 2) + beta * np.sum(Ft_ ** 2)

    rng = np.random.default_rng(8)
    for _ in range(6):
        D = rng.standard_normal(Ft.shape)
        h = 1e-5
        dd = (J(Ft + h * D) - J(Ft - h * D)) / (2 * h)
        assert abs(dd) < 1e-6 * J(Ft)


def test_calib_zero_pads_missing_rank():
    pp = S.host_probe_pairs(Np=20, m=2, d=5, L=1, rank=2, seed=9)
    P, Q, sig, _ = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.1, 4)
    assert np.all(P[0, :, 2:] == 0) and np.all(Q[0, 2:] == 0) and np.all(sig[0, 2:] == 0)


def test_rsvd_full_width_sketch_is_the_exact_fit():
    """With ell = m the sketch spans the whole error space, so the Rayleigh-Ritz step of the
    randomized fit is the exact truncated SVD of calib_fit (any q)."""
    pp = S.host_probe_pairs(Np=40, m=10, d=16, L=2, rank=10, noise=0.3, seed=21)
    Om = S.omega_matrix(16, 10, seed=21)
    P0, Q0, s0, _ = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.5, 4)
    for q in (0, 1):
        P, Q, s = O.calib_fit_rsvd(pp["E_probe"], pp["G_probe"], 0.5, 4, Om, q)
        assert _rel(s, s0) < 1e-11
        assert _rel(P, P0) < 1e-9 and _rel(Q, Q0) < 1e-9


def test_rsvd_exact_on_a_fit_of_low_rank():
    """Noise-free pairs: F_hat^T = (E^T E + beta I)^-1 E^T E M has the planted rank 3 < ell, so a
    sketch of width 5 holds its whole range and the fit equals the exact one; the two
    singular values beyond the rank are zero (zero rows of Q, zero columns of P)."""
    pp = S.host_probe_pairs(Np=60, m=20, d=24, L=2, rank=3, noise=0.0, seed=22)
    E = pp["E_probe"].astype(np.float64)
    G = np.stack([E @ pp["M"][l] for l in range(2)])  # exact rank 3 (no fp32 storage rounding)
    Om = S.omega_matrix(24, 5, seed=22)
    P0, Q0, s0, _ = O.calib_fit(E, G, 0.2, 3)
    P, Q, s = O.calib_fit_rsvd(E, G, 0.2, 5, Om, 0)
    for l in range(2):
        assert _rel(P[l, :, :3] @ Q[l, :3], P0[l] @ Q0[l]) < 1e-9
    assert _rel(s[:, :3], s0) < 1e-10
    assert np.all(s[:, 3:] == 0) and np.all(Q[:, 3:] == 0) and np.all(P[:, :, 3:] == 0)


def test_rsvd_ritz_values_interlace_and_truncation_is_near_optimal():
    """On a full-rank noisy fit: Ritz values of a projection lie below the singular values
    (sigma_i(Q_Y^T F^T) <= sigma_i(F^T)); no rank-r map beats the truncated SVD in
    Frobenius norm (Eckart-Young), and the randomized error approaches that optimum as q
    grows; Q has orthonormal rows."""
    pp = S.host_probe_pairs(Np=90, m=30, d=30, L=1, rank=6, noise=0.3, seed=23, e_scales=True)
    Om = S.omega_matrix(30, 8, seed=23)
    _, _, s_all, Fh = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.4, 30)
    r = 4
    opt = float(np.sum(s_all[0, r:] ** 2))
    errs = []
    for q in range(4):
        P, Q, s = O.calib_fit_rsvd(pp["E_probe"], pp["G_probe"], 0.4, r, Om, q)
        assert np.all(s[0] <= s_all[0, :r] * (1 + 1e-12))
        assert np.allclose(Q[0] @ Q[0].T, np.eye(r), atol=1e-12)
        err = float(np.sum((Fh[0] - P[0] @ Q[0]) ** 2))
        assert err >= opt * (1 - 1e-12)
        errs.append(err)
    assert errs[3] <= errs[0] and errs[3] <= opt * 1.01


def test_rsvd_converges_to_the_truncation_on_a_gapped_spectrum():
    """Planted rank r with little noise gives sigma_{r+1} << sigma_r; subspace iteration
    then converges like (sigma_{ell+1} / sigma_r)^(2q+1), so two power iterations already
    give the exact rank-r truncation to rounding."""
    pp = S.host_probe_pairs(Np=120, m=40, d=48, L=2, rank=4, noise=0.02, seed=24, e_scales=True)
    Om = S.omega_matrix(48, 8, seed=24)
    P0, Q0, s0, _ = O.calib_fit(pp["E_probe"], pp["G_probe"], 0.1, 4)
    P, Q, s = O.calib_fit_rsvd(pp["E_probe"], pp["G_probe"], 0.1, 4, Om, 2)
    assert _rel(s, s0) < 1e-10
    for l in range(2):
        assert _rel(P[l] @ Q[l], P0[l] @ Q0[l]) < 1e-8
    assert _rel(P, P0) < 1e-8 and _rel(Q, Q0) < 1e-8


def test_d_wide_fit_folded_through_the_head_is_the_label_space_fit():
    """Reading of the head fold: with the paper's d-wide error e = W^T eps (rows E_d = E_C W, W the
    head's C label rows, orthonormal here), the push-through identity gives
    (W^T A W + beta I)^-1 W^T = W^T (A + beta I)^-1 for A = E_C^T E_C, so F_hat_d^T = W^T F_hat_C^T:
    the d-wide fit, folded as P_C = W P_d, is the label-space fit (same beta), for the exact and
    the randomized fit alike (rank <= C <= ell)."""
    rng = np.random.default_rng(31)
    Np, C, d, L, beta = 60, 3, 24, 2, 0.3
    W = np.linalg.qr(rng.standard_normal((d, C)))[0].T  # C x d, orthonormal rows
    E_C = rng.standard_normal((Np, C))
    G = rng.standard_normal((L, Np, d))
    E_d = E_C @ W
    P_C, Q_C, s_C, _ = O.calib_fit(E_C, G, beta, C)
    P_d, Q_d, s_d, _ = O.calib_fit(E_d, G, beta, C)
    Pr, Qr, sr = O.calib_fit_rsvd(E_d, G, beta, C, S.omega_matrix(d, 5, seed=31), 0)
    for l in range(L):
        assert _rel(W @ P_d[l], P_C[l]) < 1e-10 and _rel(Q_d[l], Q_C[l]) < 1e-10
        assert _rel(W @ Pr[l], P_C[l]) < 1e-10 and _rel(Qr[l], Q_C[l]) < 1e-10
    assert _rel(s_d, s_C) < 1e-12 and _rel(sr, s_C) < 1e-12


def test_linear_network_targets_equal_backprop_gradients():
    """Check 4: on an all-linear tokenwise network h_l = W_l h_{l-1}, z = W_u h_L, the true
    hidden-state gradient is g_l = (W_L ... W_{l+1})^T W_u^T eps (S3), exactly linear in the
    head error.  Gradients are taken by central differences of the summed loss; the
    calibration fit on (eps, g_l) pairs with beta -> 0 then gives targets T_l = g_l."""
    rng = np.random.default_rng(13)
    N, d, C, Ln = 40, 5, 3, 3
    W = [rng.standard_normal((d, d)) / math.sqrt(d) for _ in range(Ln)]
    Wu = rng.standard_normal((C, d))
    h0 = rng.standard_normal((N, d))
    y = rng.integers(0, C, N)
    cols = np.arange(C)

    def forward_from(l, hl):
        h = hl
        for m in range(l, Ln):
            h = h @ W[m].T
        return h @ Wu.T

    hs = [h0]
    for m in range(Ln):
        hs.append(hs[-1] @ W[m].T)
    z = hs[-1] @ Wu.T
    E, _ = O.head_error(z, cols, y)
    grads = []
    for l in range(1, Ln + 1):
        g = np.zeros((N, d))
        h = 1e-5
        for n in range(N):
            for j in range(d):
                hp, hm = hs[l].copy(), hs[l].copy()
                hp[n, j] += h
                hm[n, j] -= h
                lp = _ce_direct(forward_from(l, hp), cols, y, np.ones(N), 0).sum()
                lm = _ce_direct(forward_from(l, hm), cols, y, np.ones(N), 0).sum()
                g[n, j] = (lp - lm) / (2 * h)
        grads.append(g)
    Gp = np.stack(grads)
    P, Q, _, _ = O.calib_fit(E, Gp, 1e-12, C)
    T, _ = O.feedback_targets(E, P, Q)
    for l in range(Ln):
        assert _rel(T[l], Gp[l]) < 1e-7


def test_alignment_special_cases():
    """The alignment cosine: 1 for gradients equal to the predictions up to a positive scale,
    -1 for the opposite direction, 0 for gradients orthogonal to every prediction (built by
    projecting the predictions' row space out), and the mean of a hand-computed per-block cosine
    otherwise; it ignores the scale of P."""
    rng = np.random.default_rng(4)
    Np, C, r, d, L = 50, 3, 2, 7, 2
    E = rng.standard_normal((Np, C))
    P = rng.standard_normal((L, C, r))
    Q = rng.standard_normal((L, r, d))
    T = np.stack([E @ P[l] @ Q[l] for l in range(L)])
    assert np.allclose(O.alignment(E, P, Q, 3.0 * T), 1.0, atol=1e-12)
    assert np.allclose(O.alignment(E, P, Q, -0.5 * T), -1.0, atol=1e-12)
    G = rng.standard_normal((L, Np, d))
    for l in range(L):
        Qo, _ = np.linalg.qr(Q[l].T)  # orthonormal basis of the rows of T_l (in R^d)
        G[l] -= (G[l] @ Qo) @ Qo.T
    assert np.allclose(O.alignment(E, P, Q, G), 0.0, atol=1e-12)
    G = rng.standard_normal((L, Np, d))
    want = [float(np.dot(G[l].ravel(), T[l].ravel()) / np.linalg.norm(G[l]) / np.linalg.norm(T[l])) for l in range(L)]
    assert np.allclose(O.alignment(E, P, Q, G), want, rtol=1e-12)
    assert np.allclose(O.alignment(E, 5.0 * P, Q, G), want, rtol=1e-12)
    assert np.all(O.alignment(E, 0.0 * P, Q, G) == 0.0)
