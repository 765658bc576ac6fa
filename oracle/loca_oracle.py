"""LoCA fp64 oracle: a plain, slow, obviously correct CPU statement of the hot path.

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check of ``__graft_entry__`` and
the ``cpu_baseline`` / reference arm of ``bench.py`` may import this module.  The CUDA
library never calls it and shares no code with it; inputs come from ``synth`` alone.

Every function follows one passage of the paper (LoCA, arXiv 2608.03020) in its order
and notation, with the paper's column-stacked matrices written token-major (one row per
token).  Notation map to the library (paper symbol -> here):

* top-layer error ``e = W_u^T (softmax(z) - onehot(y))`` (Eq. 4, Lemma in S3) -> the
  label-restricted error ``E`` (``N x C``), with ``W_u[labels]`` folded into ``P``;
* feedback map ``F_l = U_k S_k V_k^T`` (Eq. 5, S5) -> ``F_l^T = P_l Q_l`` (``C x d``);
* feedback prediction ``Q_l := F_l E`` (S3) -> targets ``T_l = E P_l Q_l`` (``N x d``);
* adapter rank ``r`` (paper) -> ``k``; feedback rank ``k`` (paper) -> ``r``;
* projected features ``p = A_l h_{l-1}`` (Eq. 1) -> rows of ``X_l A_l`` (``A_l``: ``d x k``).

Precision: fp64 throughout.  One storage step is modelled explicitly because the
GEMM that consumes ``T`` reads it in bf16: :func:`round_to_bf16` (8 significant bits,
round to nearest, ties to even) applied to ``T`` where the caller asks for it.

Parity pins: every function here is pinned by ``tests/test_oracle_pins.py`` against
closed forms, brute force, finite differences of the paper's losses, textbook library
routines or identities the paper proves.  No function is "parity unpinned".
"""

from __future__ import annotations

import numpy as np

__all__ = [
    "round_to_bf16",
    "rms",
    "head_error",
    "feedback_targets",
    "alignment",
    "scaled_step",
    "accumulate_stats",
    "project_stats",
    "kspace_stats",
    "ridge_lambdas",
    "cholesky",
    "ridge_solve",
    "calib_fit",
    "calib_fit_dual",
    "calib_fit_rsvd",
    "loca_pass",
]


def round_to_bf16(x):
    """Round to bf16 precision: 8 significant bits, round to nearest, ties to even.

    ``x = m * 2**e`` with ``0.5 <= |m| < 1`` (``frexp``); ``m * 2**8`` is rounded to the
    nearest integer with ties to even (``rint``) and scaled back.  Subnormal and
    overflow ranges of bf16 do not occur for the values this oracle rounds.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.rint(np.ldexp(m, 8)), e - 8)


def rms(X):
    """RMS(X) = ||X||_F / sqrt(a b) for a nonempty ``a x b`` matrix (S8)."""
    X = np.asarray(X, dtype=np.float64)
    return float(np.sqrt(np.sum(X * X) / X.size))


def head_error(z, label_cols, y, w=None, normaliser=0):
    """Top-layer error at the frozen head (Eq. 4; Lemma "Top-layer error", S3).

    For token ``n`` with logits ``z_n`` the cross-entropy is
    ``l_CE = -z_{n,y_n} + log sum_{j in S} exp(z_{n,j})`` and its derivative with respect
    to ``z_{n,i}`` is ``softmax_i - 1[i = y_n]``, scaled by the loss weight ``w_n``.

    The error is returned on the ``C`` label columns only (``E[n, c]`` belongs to column
    ``label_cols[c]``): ``E[n, c] = w_n (exp(z_{n, label_cols[c]} - lse_n) - 1[y_n = c])``.

    ``normaliser=0``: ``S`` is the full row (the paper's softmax over the vocabulary).
    ``normaliser=1``: ``S`` is the label columns (a softmax over the verbalizer).
    ``y_n = -1`` marks a masked position: weight 0, so ``E[n] = 0`` (S2, S3).

    Returns ``(E, ce)``: ``E`` is ``N x C``, ``ce`` the weighted per-token loss ``N``.
    """
    z = np.asarray(z, dtype=np.float64)
    cols = np.asarray(label_cols, dtype=np.int64)
    y = np.asarray(y, dtype=np.int64)
    N = z.shape[0]
    C = cols.size
    wt = np.ones(N) if w is None else np.asarray(w, dtype=np.float64).copy()
    wt[y < 0] = 0.0
    S = z if normaliser == 0 else z[:, cols]
    # log sum_{j in S} exp(z_j), evaluated with the row maximum factored out
    top = S.max(axis=1)
    lse = top + np.log(np.sum(np.exp(S - top[:, None]), axis=1))
    soft = np.exp(z[:, cols] - lse[:, None])
    onehot = (y[:, None] == np.arange(C)[None, :]).astype(np.float64)
    E = wt[:, None] * (soft - onehot)
    z_y = np.where(y >= 0, z[np.arange(N), cols[np.clip(y, 0, C - 1)]], 0.0)
    ce = wt * (lse - z_y)
    return E, ce


def feedback_targets(E, P, Q):
    """Tokenwise feedback predictions ``Q_l := F_l E`` (S3), applied through the low-rank
    factors as ``F_l e = U_k (S_k (V_k^T e))`` (S11).

    Token-major: ``T_l = (E P_l) Q_l`` with ``E`` (``N x C``), ``P_l`` (``C x r``),
    ``Q_l`` (``r x d``).  Returns ``T`` (``L x N x d``) and ``tsq[l] = ||T_l||_F^2``.
    """
    E = np.asarray(E, dtype=np.float64)
    P = np.asarray(P, dtype=np.float64)
    Q = np.asarray(Q, dtype=np.float64)
    L = P.shape[0]
    T = np.stack([(E @ P[l]) @ Q[l] for l in range(L)])
    tsq = np.array([np.sum(T[l] * T[l]) for l in range(L)])
    return T, tsq


def alignment(E, P, Q, G):
    """In-probe alignment diagnostic (supplement, "One-shot calibration": the cosine between
    the stacked feedback predictions and the stacked exact probe gradients of each block).

    ``alpha_l = <G_l, T_l>_F / (||G_l||_F ||T_l||_F)`` with ``T_l = E P_l Q_l`` (the
    predictions of :func:`feedback_targets`) and ``G_l`` (``Np x d``) the exact hidden-state
    gradients at the same probe positions.  0 where either matrix is zero.
    """
    T, tsq = feedback_targets(E, P, Q)
    G = np.asarray(G, dtype=np.float64)
    out = np.zeros(T.shape[0])
    for l in range(T.shape[0]):
        gg = float(np.sum(G[l] * G[l]))
        if gg > 0.0 and tsq[l] > 0.0:
            out[l] = float(np.sum(G[l] * T[l])) / np.sqrt(gg * tsq[l])
    return out


def scaled_step(eta, X_l, T_l):
    """Scale-normalised step (Eq. 10; S8): ``eta_bar = eta RMS(H_{l-1}) / RMS(Q_l)``,
    and ``eta_bar = 0`` when ``Q_l = 0``.  ``X_l`` is the block's adapter input for one
    mini-batch and ``T_l`` its feedback predictions for the same tokens."""
    rt = rms(T_l)
    if rt == 0.0:
        return 0.0
    return float(eta) * rms(X_l) / rt


def accumulate_stats(X_batches, T_batches, eta, t_feed=None, gram=None, cross=None, xsq_total=None):
    """Streamed sufficient statistics (Eqs. 6 and 9; S6; additivity over mini-batches, S7).

    For every mini-batch ``m`` and block ``l``:

    * ``Gram_l += X_{l,m}^T X_{l,m}`` (``d x d``; ``A_l^T Gram_l A_l`` is the paper's
      ``G_l = sum_n p p^T``);
    * ``eta_bar_{l,m}`` from :func:`scaled_step` on this batch (S8: one step per block
      and mini-batch);
    * ``Cross_l += -eta_bar_{l,m} T_{l,m}^T X_{l,m}`` (``d x d``; row = output channel,
      column = input channel), the ``-eta_bar q`` part of the residual target
      ``rho = B^(t) p - eta_bar q`` (Eq. 6) against the features, before projection;
    * ``xsq_total_l += ||X_{l,m}||_F^2`` (= trace of this batch's Gram).

    ``t_feed="bf16"`` multiplies ``X`` by ``round_to_bf16(T)`` in the cross product (the
    step itself always uses the unrounded ``T``).  Arrays are updated in place when
    given, else started at zero.  Returns ``(gram, cross, xsq_total)``.
    """
    X0 = np.asarray(X_batches[0])
    L, _, d = X0.shape
    gram = np.zeros((L, d, d)) if gram is None else gram
    cross = np.zeros((L, d, d)) if cross is None else cross
    xsq_total = np.zeros(L) if xsq_total is None else xsq_total
    for Xm, Tm in zip(X_batches, T_batches):
        Xm = np.asarray(Xm, dtype=np.float64)
        Tm = np.asarray(Tm, dtype=np.float64)
        for l in range(L):
            Xl, Tl = Xm[l], Tm[l]
            step = scaled_step(eta, Xl, Tl)
            Tf = round_to_bf16(Tl) if t_feed == "bf16" else Tl
            gram[l] += Xl.T @ Xl
            cross[l] += -step * (Tf.T @ Xl)
            xsq_total[l] += float(np.sum(Xl * Xl))
    return gram, cross, xsq_total


def project_stats(gram, cross, A, B_prev=None):
    """Project the ``d x d`` statistics onto the adapter features ``p = A_l^T x``.

    ``G_l = A_l^T Gram_l A_l`` (``k x k``; Eq. 9) and
    ``C_l = B_prev,l G_l + Cross_l A_l`` (``d x k``), which equals
    ``sum_n rho_n p_n^T`` with ``rho_n = B^(t) p_n - eta_bar q_n`` (Eqs. 6 and 9).
    ``B_prev=None`` means ``B^(t) = 0`` (the frozen model).
    """
    gram = np.asarray(gram, dtype=np.float64)
    cross = np.asarray(cross, dtype=np.float64)
    A = np.asarray(A, dtype=np.float64)
    L = A.shape[0]
    G = np.stack([A[l].T @ gram[l] @ A[l] for l in range(L)])
    C = np.stack([cross[l] @ A[l] for l in range(L)])
    if B_prev is not None:
        Bp = np.asarray(B_prev, dtype=np.float64)
        C = C + np.stack([Bp[l] @ G[l] for l in range(L)])
    return G, C


def kspace_stats(X_batches, T_batches, A, eta, B_prev=None):
    """The paper's own projected statistics, accumulated token by token over the
    mini-batches (Eq. 9; S7 additivity; S8 one step per block and mini-batch):

    ``p_n = A_l^T x_n`` (the adapter features, Eq. 1), ``rho_n = B^(t) p_n - eta_bar q_n``
    (Eq. 6, ``q_n`` the target row), ``G_l = sum_n p_n p_n^T`` (``k x k``) and
    ``C_l = sum_n rho_n p_n^T`` (``d x k``), with ``eta_bar`` from :func:`scaled_step` on the
    token's mini-batch.  Written token-major: ``P_feat = X_l A_l`` (one row per token),
    ``R = P_feat B^T - eta_bar T_l`` (rows ``rho_n^T``), ``G_l += P_feat^T P_feat``,
    ``C_l += R^T P_feat``.  The targets enter unrounded (this route never stores them).
    ``B_prev=None`` means ``B^(t) = 0``.  Returns ``(G, C, xsq_total)``.
    """
    A = np.asarray(A, dtype=np.float64)
    L, d, k = A.shape
    G = np.zeros((L, k, k))
    C = np.zeros((L, d, k))
    xsq_total = np.zeros(L)
    Bp = None if B_prev is None else np.asarray(B_prev, dtype=np.float64)
    for Xm, Tm in zip(X_batches, T_batches):
        for l in range(L):
            Xl = np.asarray(Xm[l], dtype=np.float64)
            Tl = np.asarray(Tm[l], dtype=np.float64)
            step = scaled_step(eta, Xl, Tl)
            feat = Xl @ A[l]
            R = -step * Tl
            if Bp is not None:
                R = R + feat @ Bp[l].T
            G[l] += feat.T @ feat
            C[l] += R.T @ feat
            xsq_total[l] += float(np.sum(Xl * Xl))
    return G, C, xsq_total


def ridge_lambdas(lambda_rel, xsq_total, d):
    """Ridge coefficients ``lambda_{j,l} = c_j tr(Gram_l) / d`` (``nl x L``).

    The paper requires ``lambda > 0`` and gives no value (Eq. 8); the candidate set is
    scaled by the mean per-channel energy ``tr(Gram_l)/d``.  With ``xsq_total=None`` the
    coefficients are absolute: ``lambda_{j,l} = c_j``.
    """
    c = np.asarray(lambda_rel, dtype=np.float64)
    if xsq_total is None:
        return np.repeat(c[:, None], 1, axis=1)
    return c[:, None] * np.asarray(xsq_total, dtype=np.float64)[None, :] / float(d)


def cholesky(M):
    """Lower-triangular ``L`` with ``L L^T = M`` for symmetric positive definite ``M``
    (column by column).  Returns ``(L, info)``; ``info = j + 1`` if the ``j``-th pivot is
    not positive (not positive definite), else 0."""
    M = np.asarray(M, dtype=np.float64)
    k = M.shape[0]
    Lo = np.zeros_like(M)
    for j in range(k):
        s = M[j, j] - np.dot(Lo[j, :j], Lo[j, :j])
        if not s > 0.0:
            return Lo, j + 1
        Lo[j, j] = np.sqrt(s)
        for i in range(j + 1, k):
            Lo[i, j] = (M[i, j] - np.dot(Lo[i, :j], Lo[j, :j])) / Lo[j, j]
    return Lo, 0


def ridge_solve(G, C, lam):
    """Closed-form block minimiser ``B* = C (G + lambda I)^{-1}`` (Eq. 8; Theorem S6),
    evaluated as the positive-definite system ``(G + lambda I) X = C^T``, ``B* = X^T``
    (S7), by a Cholesky factorisation and two triangular substitutions; no inverse.

    ``G``: ``L x k x k``; ``C``: ``L x d x k``; ``lam``: ``nl x L`` (or ``nl x 1``).
    Returns ``B`` (``nl x L x d x k``) and ``info`` (``nl x L``; 0 = solved).
    """
    G = np.asarray(G, dtype=np.float64)
    C = np.asarray(C, dtype=np.float64)
    lam = np.asarray(lam, dtype=np.float64)
    L, k, _ = G.shape
    d = C.shape[1]
    nl = lam.shape[0]
    B = np.zeros((nl, L, d, k))
    info = np.zeros((nl, L), dtype=np.int32)
    for j in range(nl):
        for l in range(L):
            lv = lam[j, l] if lam.shape[1] > 1 else lam[j, 0]
            Lo, inf = cholesky(G[l] + lv * np.eye(k))
            info[j, l] = inf
            if inf:
                continue
            rhs = C[l].T  # k x d
            # forward substitution  Lo Y = rhs
            Y = np.zeros_like(rhs)
            for i in range(k):
                Y[i] = (rhs[i] - Lo[i, :i] @ Y[:i]) / Lo[i, i]
            # back substitution  Lo^T Xs = Y
            Xs = np.zeros_like(rhs)
            for i in range(k - 1, -1, -1):
                Xs[i] = (Y[i] - Lo[i + 1:, i] @ Xs[i + 1:]) / Lo[i, i]
            B[j, l] = Xs.T
    return B, info


def calib_fit(E_probe, G_probe, beta, r):
    """One-shot reduced-rank feedback fit (Eq. 5; Theorem "Feedback ridge solution" and
    Lemma "Rank-truncation error", S5).

    Token-major probe pairs: ``E_probe`` (``Np x m``, rows are top errors) and
    ``G_probe[l]`` (``Np x d``, rows are exact hidden-state gradients).  The ridge fit
    ``F_hat = G E^T (E E^T + beta I)^{-1}`` (primal form) reads, transposed,
    ``F_hat^T = (E_probe^T E_probe + beta I_m)^{-1} E_probe^T G_probe[l]`` (``m x d``),
    solved as a linear system.  Its SVD ``F_hat^T = U S V^T`` is truncated to rank
    ``r``: ``P_l = U_r S_r`` (``m x r``) and ``Q_l = V_r^T`` (``r x d``), so that
    ``P_l Q_l = F_l^T``.  Ranks beyond ``min(m, d)`` are zero-padded.

    Sign convention (the SVD's signs are free): the entry of largest magnitude in each
    row of ``Q_l`` is made positive (and the matching column of ``P_l`` flipped).

    Returns ``P`` (``L x m x r``), ``Q`` (``L x r x d``), ``sigma`` (``L x r``) and
    ``F_hat_T`` (``L x m x d``, the untruncated fit).
    """
    E = np.asarray(E_probe, dtype=np.float64)
    Gp = np.asarray(G_probe, dtype=np.float64)
    L, Np, d = Gp.shape
    m = E.shape[1]
    P = np.zeros((L, m, r))
    Q = np.zeros((L, r, d))
    sig = np.zeros((L, r))
    Fh = np.zeros((L, m, d))
    lhs = E.T @ E + beta * np.eye(m)
    for l in range(L):
        Fh[l] = np.linalg.solve(lhs, E.T @ Gp[l])
        U, s, Vt = np.linalg.svd(Fh[l], full_matrices=False)
        q = min(r, s.size)
        for i in range(q):
            u, v = U[:, i].copy(), Vt[i].copy()
            if v[np.argmax(np.abs(v))] < 0:
                u, v = -u, -v
            P[l, :, i] = u * s[i]
            Q[l, i] = v
            sig[l, i] = s[i]
    return P, Q, sig, Fh


def calib_fit_dual(E_probe, G_probe, beta):
    """Dual form of the feedback ridge fit (S5, push-through identity):
    ``F_hat^T = E_probe^T (E_probe E_probe^T + beta I_Np)^{-1} G_probe[l]`` (``m x d``)."""
    E = np.asarray(E_probe, dtype=np.float64)
    Gp = np.asarray(G_probe, dtype=np.float64)
    L, Np, d = Gp.shape
    K = E @ E.T + beta * np.eye(Np)
    return np.stack([E.T @ np.linalg.solve(K, Gp[l]) for l in range(L)])


def calib_fit_rsvd(E_probe, G_probe, beta, r, Omega, q):
    """Rank-r truncation of the feedback ridge fit (Eq. 5; S5) for error spaces too wide to
    form and decompose ``F_hat_l^T`` (the paper's ``m = d`` form ``e = W_u^T eps``), by
    randomized subspace iteration: Halko, Martinsson and Tropp, "Finding structure with
    randomness" (SIAM Review 53, 2011), Algorithm 4.4 (range finder with ``q`` power
    iterations, an orthonormal basis taken after every product) followed by Algorithm 5.1
    (SVD of the matrix projected on that basis).  It approximates :func:`calib_fit`; with
    ``ell >= rank(F_hat_l^T)`` it is exact.

    ``F_hat_l^T = (E^T E + beta I_m)^{-1} E^T G_l`` (``m x d``) is only applied to blocks
    of ``ell = Omega.shape[1]`` vectors, each time by solving with ``E^T E + beta I_m``:

        F^T x = (E^T E + beta I)^{-1} E^T (G_l x),     F y = G_l^T E (E^T E + beta I)^{-1} y.

    Steps: ``Y = F^T Omega``, ``Q_Y = orth(Y)``; ``q`` times ``Z = orth(F Q_Y)``,
    ``Q_Y = orth(F^T Z)``; then ``B^T = F Q_Y`` (``d x ell``), ``B = U_B S V^T`` and
    ``U = Q_Y U_B``; ``P_l = U_r S_r``, ``Q_l = V_r^T``.  ``orth`` is any orthonormal basis
    of the columns' span (here a reduced QR).  Signs as in :func:`calib_fit` (the entry of
    largest magnitude in each ``Q_l`` row is positive); singular values at or below
    ``1e-12 sigma_1`` count as zero (zero ``Q_l`` row and ``P_l`` column).  ``Omega``
    (``d x ell``) is the caller's Gaussian test matrix, the same for every block.

    Returns ``P`` (``L x m x r``), ``Q`` (``L x r x d``) and ``sigma`` (``L x r``).
    """
    E = np.asarray(E_probe, dtype=np.float64)
    Gp = np.asarray(G_probe, dtype=np.float64)
    Om = np.asarray(Omega, dtype=np.float64)
    L, Np, d = Gp.shape
    m = E.shape[1]
    K = E.T @ E + beta * np.eye(m)

    def orth(Y):
        return np.linalg.qr(Y, mode="reduced")[0]

    P = np.zeros((L, m, r))
    Q = np.zeros((L, r, d))
    sig = np.zeros((L, r))
    for l in range(L):
        G = Gp[l]

        def Ft(X):  # F_hat^T X
            return np.linalg.solve(K, E.T @ (G @ X))

        def F(Y):  # F_hat Y
            return G.T @ (E @ np.linalg.solve(K, Y))

        QY = orth(Ft(Om))
        for _ in range(q):
            Z = orth(F(QY))
            QY = orth(Ft(Z))
        Bt = F(QY)
        UB, s, Vt = np.linalg.svd(Bt.T, full_matrices=False)
        U = QY @ UB
        for i in range(min(r, s.size)):
            if not s[i] > 1e-12 * s[0]:
                break
            u, v = U[:, i].copy(), Vt[i].copy()
            if v[np.argmax(np.abs(v))] < 0:
                u, v = -u, -v
            P[l, :, i] = u * s[i]
            Q[l, i] = v
            sig[l, i] = s[i]
    return P, Q, sig


def loca_pass(z, label_cols, y, X, P, Q, A, eta, lambda_rel, w=None, normaliser=0,
              B_prev=None, micro_batches=1, t_feed=None, relative_lambda=True):
    """One Stage-II outer iteration under a Jacobi schedule, after the forward pass
    (S13, steps 2-5; S8): head error -> feedback targets -> streamed statistics ->
    projected statistics -> positive-definite solves, for every block and every ridge
    candidate.  ``X`` is ``L x N x d``; tokens are split into ``micro_batches``
    contiguous mini-batches of ``ceil(N / micro_batches)`` tokens.

    Returns a dict with ``E, ce, T, tsq, gram, cross, xsq_total, G, C, lam, B, info``
    (``T`` and ``tsq`` over the whole pass).
    """
    E, ce = head_error(z, label_cols, y, w=w, normaliser=normaliser)
    X = np.asarray(X, dtype=np.float64)
    L, N, d = X.shape
    nb = -(-N // micro_batches)
    Xb, Tb = [], []
    for n0 in range(0, N, nb):
        n1 = min(N, n0 + nb)
        Tm, _ = feedback_targets(E[n0:n1], P, Q)
        Xb.append(X[:, n0:n1])
        Tb.append(Tm)
    gram, cross, xsq = accumulate_stats(Xb, Tb, eta, t_feed=t_feed)
    G, C = project_stats(gram, cross, A, B_prev=B_prev)
    lam = ridge_lambdas(lambda_rel, xsq if relative_lambda else None, d)
    B, info = ridge_solve(G, C, lam)
    T = np.concatenate(Tb, axis=1)
    tsq = np.array([np.sum(T[l] * T[l]) for l in range(L)])
    return dict(E=E, ce=ce, T=T, tsq=tsq, gram=gram, cross=cross, xsq_total=xsq,
                G=G, C=C, lam=lam, B=B, info=info)
