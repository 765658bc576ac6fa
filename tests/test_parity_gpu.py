"""GPU parity of every hot-path stage against the fp64 oracle, through the C ABI.

Inputs come from ``synth`` (seeded) or are drawn here with seeded numpy generators; the oracle
never sees a value the CUDA path produced.  Tolerances (each derived from the arithmetic of
the stage; see the per-test docstrings):

* error, targets (fp32): elementwise ``|gpu - ref| <= 1e-5 * scale + floor``, ``scale`` the
  magnitude sum of the terms (``|U||Q|`` for targets) or the loss weight (error);
* bf16 targets: within half a bf16 ulp of the fp64 value plus the fp32 bound above;
* Gram / cross / adapters: relative Frobenius error <= 1e-5 (fp32 inputs) and <= 2e-3
  (bf16 inputs, the bound the method's statement of the problem sets).
"""

import math
import zlib

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
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64) if t.dtype == torch.bfloat16 else \
        t.detach().cpu().numpy().astype(np.float64)


def _dev(a, dtype=torch.float32):
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


# ------------------------------------------------------------------------- error

ERROR_CASES = [
    # name, N, V, C, logit dtype, normaliser, ldz extra, masked/weighted
    ("tiny_f32", 512, 4, 4, "f32", 0, 0, False),
    ("fullrow_bf16", 777, 1531, 3, "bf16", 0, 0, True),
    ("labelnorm_bf16", 777, 1531, 3, "bf16", 1, 0, True),
    ("pitch_unaligned_bf16", 300, 999, 4, "bf16", 0, 3, True),
    ("pitch_f32", 257, 130, 2, "f32", 0, 6, False),
    ("vocab_row_bf16", 48, 151936, 4, "bf16", 0, 0, True),
    ("single_class", 64, 64, 1, "f32", 0, 0, False),
    ("wide_labels_bf16", 300, 4096, 64, "bf16", 0, 0, True),
]


@pytest.mark.parametrize("case", ERROR_CASES, ids=[c[0] for c in ERROR_CASES])
def test_error_parity(lc, case):
    """Lemma S3.  fp32 arithmetic on the GPU: a softmax entry carries ~|d lse| + 2 ulp relative
    error (1e-6 for long rows); the label entry softmax - 1 cancels, hence the absolute floor
    1e-6 * w_n."""
    name, N, V, C, ldt, normaliser, extra, mw = case
    rng = np.random.default_rng(zlib.crc32(name.encode()))
    z = rng.standard_normal((N, V)).astype(np.float32) * 2.0
    cols = np.sort(rng.choice(V, size=C, replace=False)).astype(np.int32)
    z[:, cols] += math.log(max(V / C, 1.0))
    y = rng.integers(0, C, N).astype(np.int32)
    w = None
    if mw:
        y[rng.random(N) < 0.1] = -1
        w = rng.uniform(0.25, 2.0, N).astype(np.float32)
    tdt = torch.bfloat16 if ldt == "bf16" else torch.float32
    zt = torch.zeros((N, V + extra), dtype=tdt, device="cuda")
    zt[:, :V] = _dev(z, tdt)
    zv = zt[:, :V]
    z64 = _np(zv)  # the exact logits the kernel reads (bf16-rounded inputs)
    E = torch.empty((N, C), dtype=torch.float32, device="cuda")
    ce = torch.empty((N,), dtype=torch.float32, device="cuda")
    lc.loca_error(zv, _dev(cols, torch.int32), _dev(y, torch.int32), E, w=None if w is None else _dev(w),
                  ce=ce, normaliser=normaliser)
    torch.cuda.synchronize()
    E_ref, ce_ref = O.head_error(z64, cols, y, w=w, normaliser=normaliser)
    wn = np.ones(N) if w is None else w.astype(np.float64)
    wn = np.where(y < 0, 0.0, wn)
    err = np.abs(_np(E) - E_ref)
    assert np.all(err <= 1e-5 * np.abs(E_ref) + 1e-6 * wn[:, None] + 1e-30), float(err.max())
    cerr = np.abs(_np(ce) - ce_ref)
    assert np.all(cerr <= 1e-5 * np.abs(ce_ref) + 1e-6 * wn), float(cerr.max())
    assert np.all(_np(E)[y < 0] == 0.0)


# ------------------------------------------------------------------------- targets

@pytest.mark.parametrize("tdt,L,N,d,C,r", [
    ("f32", 2, 512, 64, 4, 4),
    ("f32", 3, 1000, 328, 3, 8),
    ("f32", 2, 70, 100, 2, 5),
    ("bf16", 3, 1000, 328, 3, 8),
    ("bf16", 2, 4097, 896, 4, 16),
    ("bf16", 1, 65, 8, 1, 1),
    ("bf16", 2, 300, 512, 4, 32),
    ("f32", 1, 5000, 264, 5, 12),
    ("bf16", 1, 4100, 120, 3, 3),
    ("bf16", 2, 3000, 960, 2, 8),
    ("bf16", 1, 2000, 256, 64, 32),  # the kernel's limits: C = 64 label columns, r = 32
    ("f32", 1, 700, 136, 64, 31),
])
def test_targets_parity(lc, tdt, L, N, d, C, r):
    """S3 / S11.  Each output is an fp32 dot product of length r after an fp32 product of length C:
    |error| <= 1e-5 (|U||Q|) holds with a wide margin; bf16 output adds half an ulp."""
    rng = np.random.default_rng(N * 7 + d)
    E = rng.standard_normal((N, C)).astype(np.float32) * 0.5
    P = rng.normal(0, 1 / math.sqrt(r), (L, C, r)).astype(np.float32)
    Q = rng.normal(0, 1 / math.sqrt(r), (L, r, d)).astype(np.float32)
    tt = torch.bfloat16 if tdt == "bf16" else torch.float32
    T = torch.empty((L, N, d), dtype=tt, device="cuda")
    tsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_targets(_dev(E), _dev(P), _dev(Q), T, tsq=tsq)
    torch.cuda.synchronize()
    T_ref, tsq_ref = O.feedback_targets(E, P, Q)
    scale = np.stack([np.abs(E.astype(np.float64) @ P[l]) @ np.abs(Q[l].astype(np.float64)) for l in range(L)])
    bound = 1e-5 * scale + 1e-30
    Tg = _np(T)
    if tdt == "bf16":
        _, e = np.frexp(T_ref)
        half_ulp = np.ldexp(1.0, e - 9)  # half of 2^(e-8): bf16 keeps 8 significant bits
        bound = bound + half_ulp
    assert np.all(np.abs(Tg - T_ref) <= bound), float(np.max(np.abs(Tg - T_ref) - bound))
    assert np.allclose(_np(tsq), tsq_ref, rtol=1e-5, atol=0)


# ------------------------------------------------------------------------- accumulate

def _synthetic_stats_inputs(L, N, d, dtype, seed):
    rng = np.random.default_rng(seed)
    s = rng.lognormal(0, 0.5, (L, 1, d))
    X = (rng.standard_normal((L, N, d)) * s).astype(np.float32)
    T = (rng.standard_normal((L, N, d)) * 0.05).astype(np.float32)
    if dtype == "bf16":
        X = torch.from_numpy(X).to(torch.bfloat16).float().numpy()
        T = torch.from_numpy(T).to(torch.bfloat16).float().numpy()
    return X.astype(np.float64), T.astype(np.float64)


@pytest.mark.parametrize("dtype,L,d,batches", [
    ("f32", 2, 64, (512,)),
    ("f32", 2, 72, (300, 41)),
    ("bf16", 2, 328, (1000, 77)),
    ("bf16", 1, 64, (64,)),
    ("bf16", 3, 8, (1, 5)),
    ("bf16", 2, 896, (4096,)),
    ("bf16", 1, 1536, (640, 640)),
    ("bf16", 2, 640, (40000, 17000)),  # several accumulation segments, ragged; then accumulate
])
def test_accumulate_parity(lc, dtype, L, d, batches):
    """Eqs. 6, 9, 10; S7, S8.  fp32 inputs: fp64 accumulation, one fp32 rounding -> 1e-5 holds
    with margin.  bf16 inputs: bf16 products are exact in fp32 and the tensor core accumulates
    in fp32, so the error is that of fp32 summation over N tokens (<< 2e-3)."""
    eta = 0.01
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    gram = torch.empty((L, d, d), dtype=torch.float32, device="cuda")
    cross = torch.empty_like(gram)
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    Xs, Ts = [], []
    for b, n in enumerate(batches):
        X, T = _synthetic_stats_inputs(L, n, d, dtype, seed=1000 * b + d)
        Xs.append(X)
        Ts.append(T)
        tsq = _dev(np.array([np.sum(T[l] ** 2) for l in range(L)]), torch.float64)
        lc.loca_accumulate(_dev(X, tdt), _dev(T, tdt), tsq, eta, gram, cross, xsq, zero_first=(b == 0))
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    g_ref, c_ref, x_ref = O.accumulate_stats(Xs, Ts, eta)
    tol = 1e-5 if dtype == "f32" else 2e-3
    rg, rc = _rel(_np(gram), g_ref), _rel(_np(cross), c_ref)
    print(f"rel err gram {rg:.3e} cross {rc:.3e}")
    assert rg <= tol and rc <= tol
    # f32 path: fp64 sums (1e-12).  bf16 path: exact squares summed in fp32 partials of at most
    # 32 terms, partials summed in fp64: relative error <= 32 * 2^-24 < 2e-6.
    assert np.allclose(_np(xsq), x_ref, rtol=1e-12 if dtype == "f32" else 2e-6, atol=0)
    gg = _np(gram)
    assert np.array_equal(gg, np.transpose(gg, (0, 2, 1)))  # both halves written, identical
    if dtype == "bf16":
        # bf16 inputs are exact; the only error is fp32 accumulation: far inside 2e-3
        assert rg <= 1e-4 and rc <= 1e-4


def test_gram_accumulation_bias_is_bounded_over_long_batches(lc):
    """Eq. 9 and S7 ask for exact sums.  The tensor cores accumulate in fp32 and lose a fraction of
    an ulp of the running sum toward zero at every MMA step (K = 16 tokens), so an accumulator fed
    N tokens drifts by about N/16 such losses relative to its value: 6.5e-4 at 131072 tokens.  The
    kernel restarts its accumulators every 16384 tokens and adds the segments into the fp32 output
    with round-to-nearest additions, so the drift no longer grows with N.  At 2^20 tokens in one
    call: Gram, cross product and the Gram trace (= ||X||^2) within 1e-4 of the fp64 sums."""
    L, N, d = 1, 1 << 20, 512
    X, T = _synthetic_stats_inputs(L, N, d, "bf16", seed=77)
    Xd, Td = _dev(X, torch.bfloat16), _dev(T, torch.bfloat16)
    gram = torch.empty((L, d, d), dtype=torch.float32, device="cuda")
    cross = torch.empty_like(gram)
    tsq = _dev(np.array([np.sum(T[l] ** 2) for l in range(L)]), torch.float64)
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    alpha = torch.empty((L,), dtype=torch.float32, device="cuda")
    lc.loca_gram_cross(Xd, Td, torch.ones((L,), dtype=torch.float32, device="cuda"), gram, cross, zero_first=True)
    lc.loca_step_from_gram(gram, tsq, 0.01, xsq, alpha)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    del Xd, Td
    g_ref = X[0].T @ X[0]
    c_ref = T[0].T @ X[0]
    rg, rc = _rel(_np(gram[0]), g_ref), _rel(_np(cross[0]), c_ref)
    tr = float(np.trace(g_ref))
    rx = (float(xsq[0]) - tr) / tr
    print(f"N = 2^20: rel err gram {rg:.2e} cross {rc:.2e} trace {rx:+.2e}")
    assert rg <= 1e-4 and rc <= 1e-4 and abs(rx) <= 1e-4


def test_accumulate_deterministic(lc):
    L, N, d = 2, 2000, 392
    X, T = _synthetic_stats_inputs(L, N, d, "bf16", seed=5)
    Xd, Td = _dev(X, torch.bfloat16), _dev(T, torch.bfloat16)
    tsq = _dev(np.array([np.sum(T[l] ** 2) for l in range(L)]), torch.float64)
    outs = []
    for _ in range(2):
        gram = torch.empty((L, d, d), dtype=torch.float32, device="cuda")
        cross = torch.empty_like(gram)
        xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
        lc.loca_accumulate(Xd, Td, tsq, 0.03, gram, cross, xsq, zero_first=True)
        outs.append((gram.clone(), cross.clone(), xsq.clone()))
    torch.cuda.synchronize()
    for a, b in zip(outs[0], outs[1]):
        assert torch.equal(a, b)


def test_accumulate_empty_batch_zeroes(lc):
    L, d = 2, 64
    gram = torch.full((L, d, d), 3.0, device="cuda")
    cross = torch.full((L, d, d), 3.0, device="cuda")
    xsq = torch.full((L,), 7.0, dtype=torch.float64, device="cuda")
    X = torch.empty((L, 0, d), dtype=torch.bfloat16, device="cuda")
    tsq = torch.zeros((L,), dtype=torch.float64, device="cuda")
    lc.loca_accumulate(X, X, tsq, 0.01, gram, cross, xsq, zero_first=True)
    torch.cuda.synchronize()
    assert torch.count_nonzero(gram) == 0 and torch.count_nonzero(cross) == 0 and torch.count_nonzero(xsq) == 0


def test_zero_targets_give_zero_cross(lc):
    L, N, d = 1, 256, 64
    X, _ = _synthetic_stats_inputs(L, N, d, "bf16", seed=9)
    T = np.zeros((L, N, d))
    gram = torch.empty((L, d, d), device="cuda")
    cross = torch.empty_like(gram)
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_accumulate(_dev(X, torch.bfloat16), _dev(T, torch.bfloat16), torch.zeros(L, dtype=torch.float64,
                       device="cuda"), 0.01, gram, cross, xsq, zero_first=True)
    torch.cuda.synchronize()
    assert torch.count_nonzero(cross) == 0


@pytest.mark.parametrize("dtype,L,N,d,group,host", [
    ("bf16", 5, 1000, 328, 2, "loca"),
    ("bf16", 3, 2048, 512, 1, "pageable"),
    ("bf16", 4, 700, 896, 4, "torch"),
    ("f32", 3, 300, 72, 2, "loca"),
])
def test_accumulate_streamed_matches_device_path(lc, dtype, L, N, d, group, host):
    """Eqs. 6, 9, 10; S7.  X streamed from host memory in groups of blocks gives the statistics of
    the device-resident call: Gram and cross bit for bit where each block's step is the same
    (the kernels of one block do not depend on the other blocks), xsq / alpha to the rounding of
    a differently split fp64 sum.  Two calls in a row (overwrite, then accumulate) also exercise
    the reuse of the two staging slots across calls; checked against the oracle as well."""
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    eta = 0.02
    Xs, Ts, ref, got, hosts = [], [], [], [], []
    staging = torch.empty((2 * group, N, d), dtype=tdt, device="cuda")
    for rep in range(2):
        X, T = _synthetic_stats_inputs(L, N, d, dtype, seed=77 + rep + d)
        Xs.append(X)
        Ts.append(T)
        Xd, Td = _dev(X, tdt), _dev(T, tdt)
        tsq = _dev(np.array([np.sum(T[l] ** 2) for l in range(L)]), torch.float64)
        Xh = Xd.cpu()
        if host == "torch":
            Xh = Xh.pin_memory()
        elif host == "loca":
            Xh = lc.host_empty(Xh.shape, Xh.dtype).copy_(Xh)
        hosts.append(Xh)  # host memory must outlive the copies the call queues
        # device-resident reference call and streamed call, each continuing its own accumulators
        if rep == 0:
            dg = torch.empty((L, d, d), device="cuda"); dc = torch.empty_like(dg)
            dx = torch.empty((L,), dtype=torch.float64, device="cuda")
            sg = torch.empty_like(dg); sc = torch.empty_like(dg); sx = torch.empty_like(dx)
            ref.append((dg, dc, dx))
            got.append((sg, sc, sx))
        dg, dc, dx = ref[0]
        sg, sc, sx = got[0]
        lc.loca_accumulate(Xd, Td, tsq, eta, dg, dc, dx, zero_first=(rep == 0))
        lc.loca_accumulate_streamed(Xh, staging, Td, tsq, eta, sg, sc, sx, zero_first=(rep == 0), group=group)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    dg, dc, dx = ref[0]
    sg, sc, sx = got[0]
    assert torch.equal(sg, dg)
    tol = 1e-6
    assert _rel(_np(sc), _np(dc)) <= tol
    assert np.allclose(_np(sx), _np(dx), rtol=1e-12, atol=0)
    g_ref, c_ref, x_ref = O.accumulate_stats(Xs, Ts, eta)
    t = 1e-5 if dtype == "f32" else 2e-3
    assert _rel(_np(sg), g_ref) <= t and _rel(_np(sc), c_ref) <= t


def test_host_empty_is_pinned_zeroed_and_freed(lc):
    """loca_host_alloc memory: page-locked (device-visible), zero-filled, rounded to 2 MiB, and
    released when the last tensor viewing it goes away (allocating again reuses the space)."""
    import gc

    for _ in range(3):
        h = lc.host_empty((3, 1000, 333), torch.bfloat16)
        assert h.is_pinned() and h.shape == (3, 1000, 333)
        assert torch.count_nonzero(h) == 0
        v = h[1]
        del h
        gc.collect()
        v.fill_(2.0)  # the view keeps the allocation alive
        d = v.to("cuda", non_blocking=True)
        torch.cuda.synchronize()
        assert float(d.float().sum()) == 2.0 * 1000 * 333
        del v, d
        gc.collect()
    assert lc.host_empty((0, 5), torch.float32).numel() == 0


# ------------------------------------------------------------------------- ridge solve

@pytest.mark.parametrize("k,d,L,with_prev,relative", [
    (4, 64, 2, False, True),
    (8, 200, 3, True, True),
    (16, 328, 2, True, False),
    (32, 96, 2, False, True),
    (32, 520, 2, True, True),
    (1, 16, 1, True, True),
])
def test_ridge_solve_parity(lc, k, d, L, with_prev, relative):
    """Eq. 8 / Theorem S6 stage-wise: the oracle's statistics, rounded to fp32, feed both sides.
    fp32 projections over d terms and an fp64 factorisation: 1e-5 relative Frobenius."""
    rng = np.random.default_rng(k * 100 + d)
    N = 3 * d
    X = rng.standard_normal((L, N, d)) * rng.lognormal(0, 0.5, (L, 1, d))
    T = rng.standard_normal((L, N, d)) * 0.1
    g, c, xs = O.accumulate_stats([X], [T], 0.01)
    g32 = g.astype(np.float32)
    c32 = c.astype(np.float32)
    A = np.stack([np.linalg.qr(rng.standard_normal((d, k)))[0] for _ in range(L)]).astype(np.float32)
    Bp = (0.01 * rng.standard_normal((L, d, k))).astype(np.float32) if with_prev else None
    lam_rel = [1e-4, 1e-3, 1e-2] if relative else [0.5, 50.0]
    G_ref, C_ref = O.project_stats(g32, c32, A, B_prev=Bp)
    lam = O.ridge_lambdas(lam_rel, xs if relative else None, d)
    B_ref, info_ref = O.ridge_solve(G_ref, C_ref, lam)
    nl = len(lam_rel)
    B = torch.empty((nl, L, d, k), device="cuda")
    info = torch.empty((nl, L), dtype=torch.int32, device="cuda")
    Gout = torch.empty((L, k, k), device="cuda")
    Cout = torch.empty((L, d, k), device="cuda")
    lc.loca_ridge_solve(_dev(g32), _dev(c32), _dev(A), lam_rel, B, info,
                        xsq_total=_dev(xs, torch.float64) if relative else None,
                        B_prev=None if Bp is None else _dev(Bp), G_out=Gout, C_out=Cout)
    torch.cuda.synchronize()
    assert np.array_equal(info.cpu().numpy(), info_ref)
    assert _rel(_np(Gout), G_ref) < 1e-5
    assert _rel(_np(Cout), C_ref) < 1e-5
    for j in range(nl):
        for l in range(L):
            assert _rel(_np(B)[j, l], B_ref[j, l]) < 1e-5, (j, l)


@pytest.mark.parametrize("k,d,L", [
    (16, 3584, 2),   # the 7B width: tensor-core projection, 28 row tiles and 112 K-slabs per matrix
    (32, 5120, 1),   # the 14B width (k = 32)
    (12, 1000, 2),   # k padded to 16, a ragged last row tile (104 rows) and a ragged last K-slab
    (20, 640, 3),    # k padded to 32 (N = 96 with zero columns), five row tiles per matrix
    (28, 1152, 1),   # k padded to 32, nine row tiles, 36 K-slabs
    (6, 330, 2),     # k % 4 != 0 and d % 4 != 0: the SIMT projection
])
def test_ridge_solve_parity_at_full_width(lc, k, d, L):
    """Eq. 9 projections and Theorem S6 solves at the widths of the headline workloads: the Gram
    stand-in is X^T X + diag over 256 rows with LogNormal channel scales (positive definite), the
    cross product dense; 1e-5 relative Frobenius on G = A^T Gram A, C = B_prev G + Cross A and B."""
    rng = np.random.default_rng(k + d)
    Y = rng.standard_normal((L, 256, d)) * rng.lognormal(0, 0.5, (L, 1, d))
    g = np.transpose(Y, (0, 2, 1)) @ Y
    g[:, np.arange(d), np.arange(d)] += rng.uniform(0.5, 2.0, (L, d))
    c = 0.1 * rng.standard_normal((L, d, d)) * rng.lognormal(0, 0.5, (L, 1, d))
    g32, c32 = g.astype(np.float32), c.astype(np.float32)
    xs = np.trace(g32.astype(np.float64), axis1=1, axis2=2)
    A = np.stack([np.linalg.qr(rng.standard_normal((d, k)))[0] for _ in range(L)]).astype(np.float32)
    Bp = (0.01 * rng.standard_normal((L, d, k))).astype(np.float32)
    lam_rel = [1e-4, 1e-2]
    G_ref, C_ref = O.project_stats(g32, c32, A, B_prev=Bp)
    B_ref, info_ref = O.ridge_solve(G_ref, C_ref, O.ridge_lambdas(lam_rel, xs, d))
    B = torch.empty((2, L, d, k), device="cuda")
    info = torch.empty((2, L), dtype=torch.int32, device="cuda")
    Gout = torch.empty((L, k, k), device="cuda")
    Cout = torch.empty((L, d, k), device="cuda")
    lc.loca_ridge_solve(_dev(g32), _dev(c32), _dev(A), lam_rel, B, info, xsq_total=_dev(xs, torch.float64),
                        B_prev=_dev(Bp), G_out=Gout, C_out=Cout)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    assert np.array_equal(info.cpu().numpy(), info_ref)
    eg, ec = _rel(_np(Gout), G_ref), _rel(_np(Cout), C_ref)
    eb = max(_rel(_np(B)[j, l], B_ref[j, l]) for j in range(2) for l in range(L))
    print(f"k={k} d={d}: rel err G {eg:.2e} C {ec:.2e} B {eb:.2e}")
    assert eg < 1e-5 and ec < 1e-5 and eb < 1e-5


def test_ridge_solve_reports_not_positive_definite(lc):
    L, d, k = 1, 32, 4
    g = -np.eye(d, dtype=np.float32)[None] * 100.0
    c = np.ones((L, d, d), dtype=np.float32)
    A = np.eye(d, k, dtype=np.float32)[None]
    B = torch.full((1, L, d, k), 5.0, device="cuda")
    info = torch.empty((1, L), dtype=torch.int32, device="cuda")
    lc.loca_ridge_solve(_dev(g), _dev(c), _dev(A), [1.0], B, info)
    torch.cuda.synchronize()
    assert info.item() == 1
    assert torch.count_nonzero(B) == 0


# ------------------------------------------------------------------------- end to end

def _run_pass(lc, w, f, X_host, B_prev=None, batches=1):
    act = torch.bfloat16 if w.act_dtype == "bf16" else torch.float32
    ps = lc.Pass(w.L, w.N, w.d, w.C, w.r, w.k, act, w.lambda_rel, w.eta, micro_batches=batches)
    nb = -(-w.N // batches)
    Xd = [_dev(X_host[:, n0:n0 + nb], act) for n0 in range(0, w.N, nb)]
    ps.run(_dev(f["z"]), _dev(f["label_cols"], torch.int32), _dev(f["y"], torch.int32),
           Xd if batches > 1 else Xd[0], _dev(f["P"]), _dev(f["Q"]), _dev(f["A"]),
           B_prev=None if B_prev is None else _dev(B_prev))
    torch.cuda.synchronize()
    return ps


def test_end_to_end_tiny_f32(lc):
    """The tiny workload (fp32): every output of the pass within 1e-5 of the oracle."""
    w = S.WORKLOADS["tiny"]
    f = S.host_inputs(w)
    X = f["X"].astype(np.float64)
    ps = _run_pass(lc, w, f, f["X"])
    ref = O.loca_pass(f["z"], f["label_cols"], f["y"], X, f["P"], f["Q"], f["A"], w.eta, w.lambda_rel)
    assert _rel(_np(ps.E), ref["E"]) < 1e-5
    assert _rel(_np(ps.gram), ref["gram"]) < 1e-5
    assert _rel(_np(ps.cross), ref["cross"]) < 1e-5
    assert np.allclose(_np(ps.xsq), ref["xsq_total"], rtol=1e-12)
    assert np.all(ps.info.cpu().numpy() == 0)
    assert _rel(_np(ps.B), ref["B"]) < 1e-5


@pytest.mark.parametrize("batches,prev", [(1, False), (3, True)])
def test_end_to_end_bf16_small(lc, batches, prev):
    """A scaled-down bf16 workload spanning several tensor-core tiles with ragged edges: the
    oracle rounds T to bf16 for the cross product as the GEMM feed does; B within 2e-3."""
    w = S.scaled(S.WORKLOADS["qwen2.5-0.5b"], L=3, d=392, N=1500, C=3, V=3, r=8, k=8)
    f = S.host_inputs(w)
    Bp = S.host_B_prev(w) if prev else None
    ps = _run_pass(lc, w, f, f["X"], B_prev=Bp, batches=batches)
    ref = O.loca_pass(f["z"], f["label_cols"], f["y"], f["X"].astype(np.float64), f["P"], f["Q"], f["A"], w.eta,
                      w.lambda_rel, B_prev=Bp, micro_batches=batches, t_feed="bf16")
    rg = _rel(_np(ps.gram), ref["gram"])
    rc = _rel(_np(ps.cross), ref["cross"])
    rb = max(_rel(_np(ps.B)[j, l], ref["B"][j, l]) for j in range(len(w.lambda_rel)) for l in range(w.L))
    print(f"rel err gram {rg:.2e} cross {rc:.2e} B {rb:.2e}")
    assert rg < 2e-3 and rc < 2e-3 and rb < 2e-3
    assert np.allclose(_np(ps.xsq), ref["xsq_total"], rtol=2e-6)
    assert lc.loca_device_status() == 0


def _single_batch_chain(lc, w, f, X, Bp=None):
    """error -> targets -> Gram / cross at alpha = 1 -> step from the Gram trace -> solve with
    cross_scale = alpha: the pass with one mini-batch that reads X once (in the Gram kernel)."""
    act = torch.bfloat16 if w.act_dtype == "bf16" else torch.float32
    L, N, d, C, r, k = w.L, w.N, w.d, w.C, w.r, w.k
    nl = len(w.lambda_rel)
    f32 = dict(device="cuda", dtype=torch.float32)
    E = torch.empty((N, C), **f32)
    T = torch.empty((L, N, d), device="cuda", dtype=act)
    tsq = torch.empty((L,), device="cuda", dtype=torch.float64)
    xsq = torch.empty((L,), device="cuda", dtype=torch.float64)
    alpha = torch.empty((L,), **f32)
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    B = torch.empty((nl, L, d, k), **f32)
    info = torch.empty((nl, L), device="cuda", dtype=torch.int32)
    C_out = torch.empty((L, d, k), **f32)
    lc.loca_error(_dev(f["z"]), _dev(f["label_cols"], torch.int32), _dev(f["y"], torch.int32), E)
    lc.loca_targets(E, _dev(f["P"]), _dev(f["Q"]), T, tsq=tsq)
    lc.loca_gram_cross(_dev(X, act), T, torch.ones((L,), **f32), gram, cross, zero_first=True)
    lc.loca_step_from_gram(gram, tsq, w.eta, xsq, alpha)
    lc.loca_ridge_solve(gram, cross, _dev(f["A"]), w.lambda_rel, B, info, xsq_total=xsq,
                        B_prev=None if Bp is None else _dev(Bp), C_out=C_out, cross_scale=alpha)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0 and int(info.abs().sum()) == 0
    return dict(xsq=_np(xsq), alpha=_np(alpha), B=_np(B), C=_np(C_out), cross=_np(cross), gram=_np(gram), tsq=_np(tsq))


@pytest.mark.parametrize("prev", [False, True])
def test_single_batch_chain_bf16(lc, prev):
    """The one-mini-batch chain (step from tr(Gram), alpha applied in the solve) against the
    oracle's pass: B and C within 2e-3, the unscaled cross product is T^T X (bf16 feed), and
    alpha / xsq agree with the separate sum-of-squares step."""
    w = S.scaled(S.WORKLOADS["qwen2.5-0.5b"], L=3, d=392, N=1500, C=3, V=3, r=8, k=8)
    f = S.host_inputs(w)
    Bp = S.host_B_prev(w) if prev else None
    out = _single_batch_chain(lc, w, f, f["X"], Bp)
    ref = O.loca_pass(f["z"], f["label_cols"], f["y"], f["X"].astype(np.float64), f["P"], f["Q"], f["A"], w.eta,
                      w.lambda_rel, B_prev=Bp, t_feed="bf16")
    assert np.allclose(out["xsq"], ref["xsq_total"], rtol=1e-5)
    alpha_ref = -w.eta * np.sqrt(ref["xsq_total"] / ref["tsq"])
    assert np.allclose(out["alpha"], alpha_ref, rtol=1e-5)
    assert _rel(out["cross"] * out["alpha"][:, None, None], ref["cross"]) < 2e-3
    assert _rel(out["C"], ref["C"]) < 2e-3
    rb = max(_rel(out["B"][j, l], ref["B"][j, l]) for j in range(len(w.lambda_rel)) for l in range(w.L))
    assert rb < 2e-3, rb
    # the separate step on the same inputs gives the same alpha
    X = _dev(f["X"], torch.bfloat16)
    xsq2 = torch.empty((w.L,), device="cuda", dtype=torch.float64)
    alpha2 = torch.empty((w.L,), device="cuda")
    lc.loca_batch_step(X, _dev(out["tsq"], torch.float64), w.eta, xsq2, alpha2, True)
    torch.cuda.synchronize()
    assert np.allclose(out["alpha"], _np(alpha2), rtol=1e-5)


def test_single_batch_chain_f32_tiny(lc):
    """The same chain on the fp32 tiny workload: B within 1e-5 of the oracle (the trace is read
    from the fp32-stored Gram diagonal, ~1e-7 relative)."""
    w = S.WORKLOADS["tiny"]
    f = S.host_inputs(w)
    out = _single_batch_chain(lc, w, f, f["X"])
    ref = O.loca_pass(f["z"], f["label_cols"], f["y"], f["X"].astype(np.float64), f["P"], f["Q"], f["A"], w.eta,
                      w.lambda_rel)
    assert np.allclose(out["xsq"], ref["xsq_total"], rtol=1e-6)
    assert _rel(out["B"], ref["B"]) < 1e-5


def test_step_from_gram_with_zero_targets(lc):
    """tsq = 0 (zero feedback, T = 0): the step is 0 (Eq. 10's convention), the trace still gives
    ||X||^2, and the solve with that cross_scale leaves C = B_prev G."""
    L, N, d, k = 2, 512, 128, 8
    X, _ = _synthetic_stats_inputs(L, N, d, "bf16", seed=10)
    Xd = _dev(X, torch.bfloat16)
    gram = torch.empty((L, d, d), device="cuda")
    cross = torch.empty_like(gram)
    lc.loca_gram_cross(Xd, torch.zeros_like(Xd), torch.ones((L,), device="cuda"), gram, cross, zero_first=True)
    tsq = torch.zeros((L,), dtype=torch.float64, device="cuda")
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    alpha = torch.full((L,), 7.0, device="cuda")
    lc.loca_step_from_gram(gram, tsq, 0.01, xsq, alpha)
    A = _dev(np.linalg.qr(np.random.default_rng(3).standard_normal((d, k)))[0][None].repeat(L, 0))
    Bp = _dev(0.01 * np.random.default_rng(4).standard_normal((L, d, k)))
    B = torch.empty((1, L, d, k), device="cuda")
    info = torch.empty((1, L), dtype=torch.int32, device="cuda")
    G_out = torch.empty((L, k, k), device="cuda")
    C_out = torch.empty((L, d, k), device="cuda")
    lc.loca_ridge_solve(gram, cross, A, [1e-3], B, info, xsq_total=xsq, B_prev=Bp, G_out=G_out, C_out=C_out,
                        cross_scale=alpha)
    torch.cuda.synchronize()
    assert torch.count_nonzero(alpha) == 0
    x64 = X.astype(np.float64)
    assert np.allclose(_np(xsq), (x64 ** 2).sum(axis=(1, 2)), rtol=1e-5)
    C_ref = np.einsum("ldk,lkj->ldj", _np(Bp).astype(np.float64), _np(G_out).astype(np.float64))
    assert _rel(_np(C_out), C_ref) < 1e-5
