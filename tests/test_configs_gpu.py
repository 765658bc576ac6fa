"""Parity at every synthetic workload's own shape, in the launch configuration ``bench.py`` times.

Each workload of ``synth.WORKLOADS`` (the paper's Qwen2.5 0.5B / 1.5B / 7B / 14B and SmolLM2-1.7B
shapes) runs through the C ABI at full size: all L blocks, all N tokens, the full logit row.  The
fp64 oracle then recomputes the chain for the first and the last block over all N tokens and every
output of those blocks is compared:

* head error ``E`` and loss ``ce``: every token, element by element (at V >> C the oracle's
  full-row softmax runs over row chunks on host threads);
* targets ``T``: every element of both blocks (bf16: half an ulp plus the fp32 bound);
* ``||T_l||^2``, ``||X_l||^2``, the step, Gram, cross product, ``G``, ``C`` and every adapter ``B``.

Single-batch workloads take the bench's chain (cross product at alpha = 1, the step from the Gram
trace, alpha applied in the solve); the 1.5B workload streams 8 micro-batches of 8192 tokens
through ``loca_targets`` + ``loca_accumulate`` with one step per batch (S7, S8).  Where the bench
also times the paper's own k-space statistics, they run on the same inputs and are checked
against the oracle's per-token statistics (``kspace_stats``).  The scale-reuse check of the
SmolLM2 row (Prop. S8 with lambda proportional to tr(Gram)/d) runs the same candidate set on X
and on a X.
"""

import concurrent.futures as cf

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
    if t.dtype == torch.float64:
        return t.detach().cpu().numpy()
    return t.detach().float().cpu().numpy().astype(np.float64)


def _rel(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _free():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


# ----------------------------------------------------------------------------- oracle side

def _oracle_error(z, cols, y, rows_per_chunk=512, threads=8):
    """The oracle's head error over every row of the device logits ``z``: rows are copied to the
    host in chunks and each chunk goes through ``O.head_error`` (a row's arithmetic is its own, so
    chunking rows changes nothing) on a pool of host threads."""
    N = z.shape[0]
    y_h = y.cpu().numpy()
    cols_h = cols.cpu().numpy()

    def one(n0):
        n1 = min(N, n0 + rows_per_chunk)
        zc = z[n0:n1].float().cpu().numpy()
        return O.head_error(zc, cols_h, y_h[n0:n1])

    with cf.ThreadPoolExecutor(max_workers=threads) as ex:
        parts = list(ex.map(one, range(0, N, rows_per_chunk)))
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def _oracle_block(E_ref, X_h, f, l, w, micro_batches=1, kspace=False):
    """The oracle chain for block ``l`` (the sequence of ``O.loca_pass`` after its head error):
    targets, streamed statistics with one step per mini-batch, projection, lambdas, solves."""
    N = X_h.shape[1]
    nb = -(-N // micro_batches)
    P, Q, A = f["P"][l:l + 1], f["Q"][l:l + 1], f["A"][l:l + 1]
    Xb, Tb = [], []
    for n0 in range(0, N, nb):
        n1 = min(N, n0 + nb)
        Tm, _ = O.feedback_targets(E_ref[n0:n1], P, Q)
        Xb.append(X_h[:, n0:n1])
        Tb.append(Tm)
    gram, cross, xsq = O.accumulate_stats(Xb, Tb, w.eta, t_feed="bf16" if w.act_dtype == "bf16" else None)
    G, C = O.project_stats(gram, cross, A)
    lam = O.ridge_lambdas(w.lambda_rel, xsq, w.d)
    B, info = O.ridge_solve(G, C, lam)
    T = np.concatenate(Tb, axis=1)
    out = dict(T=T, tsq=np.array([np.sum(T[0] * T[0])]), gram=gram, cross=cross, xsq_total=xsq, G=G, C=C, B=B,
               info=info, steps=[O.scaled_step(w.eta, Xm[0], Tm[0]) for Xm, Tm in zip(Xb, Tb)])
    if kspace:
        Gk, Ck, xk = O.kspace_stats(Xb, Tb, A, w.eta)
        Bk, infok = O.ridge_solve(Gk, Ck, O.ridge_lambdas(w.lambda_rel, xk, w.d))
        out.update(Gk=Gk, Ck=Ck, Bk=Bk, infok=infok)
    return out


# ----------------------------------------------------------------------------- comparisons

def _check_error(E, ce, E_ref, ce_ref):
    """Lemma S3 in fp32: a softmax entry carries ~1e-6 relative error over a long row; the label
    entry softmax - 1 cancels, hence the absolute floor 1e-6 of the (unit) loss weight."""
    Eg, cg = _np(E), _np(ce)
    err = np.abs(Eg - E_ref)
    assert np.all(err <= 1e-5 * np.abs(E_ref) + 1e-6), float(err.max())
    cerr = np.abs(cg - ce_ref)
    assert np.all(cerr <= 1e-5 * np.abs(ce_ref) + 1e-6), float(cerr.max())


def _check_targets(T_dev, T_ref, E_ref, P, Q, chunk=16384):
    """Every element: half a bf16 ulp (one rounding of the fp32 product) plus the fp32 bound of
    the products relative to the magnitude sum (|E| |P|) |Q|, plus the head error's own absolute
    error (<= 1e-6 per entry, carried through |P| |Q|)."""
    Pa = np.abs(P.astype(np.float64))
    Qa = np.abs(Q.astype(np.float64))
    e_abs = (np.ones((1, Pa.shape[0])) @ Pa) @ Qa
    bf16 = T_dev.dtype == torch.bfloat16
    worst = -np.inf
    for n0 in range(0, T_ref.shape[0], chunk):
        n1 = min(T_ref.shape[0], n0 + chunk)
        Tg = _np(T_dev[n0:n1])
        Tr = T_ref[n0:n1]
        scale = (np.abs(E_ref[n0:n1]) @ Pa) @ Qa
        bound = 1e-5 * scale + 1e-6 * e_abs + 1e-30
        if bf16:
            _, e = np.frexp(Tr)
            bound = bound + np.ldexp(1.0, e - 9)
        worst = max(worst, float(np.max(np.abs(Tg - Tr) - bound)))
    assert worst <= 0.0, worst


def _check_stats(tag, gram_g, cross_g, B_g, ref, nl):
    gg = _np(gram_g)
    cg = _np(cross_g)
    assert np.array_equal(gg, gg.T), f"{tag}: Gram not symmetric"
    rg, rc = _rel(gg, ref["gram"][0]), _rel(cg, ref["cross"][0])
    rb = [_rel(_np(B_g[j]), ref["B"][j, 0]) for j in range(nl)]
    print(f"{tag}: rel err gram {rg:.2e} cross {rc:.2e} B {' '.join(f'{v:.2e}' for v in rb)}")
    assert rg <= 2e-3 and rc <= 2e-3 and max(rb) <= 2e-3
    # the same drift bound as the trace: the segmented accumulation keeps the statistics well
    # inside the bf16 tolerance at every workload size
    assert rg <= 2e-4 and rc <= 2e-4


# ----------------------------------------------------------------------------- single batch

def _device_chain(lc, w, inp):
    """The bench's step: error -> targets -> Gram / cross at alpha = 1 -> step from tr(Gram) ->
    solve with alpha as cross_scale; plus the separate step of Eq. 10 from an fp64 sum of squares."""
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, k = w.L, w.N, w.d, w.C, w.k
    nl = len(w.lambda_rel)
    dev = X.device
    f32 = dict(dtype=torch.float32, device=dev)
    o = dict(E=torch.empty((N, C), **f32), ce=torch.empty((N,), **f32),
             T=torch.empty((L, N, d), dtype=X.dtype, device=dev),
             tsq=torch.empty((L,), dtype=torch.float64, device=dev),
             xsq=torch.empty((L,), dtype=torch.float64, device=dev), alpha=torch.empty((L,), **f32),
             gram=torch.empty((L, d, d), **f32), cross=torch.empty((L, d, d), **f32),
             B=torch.empty((nl, L, d, k), **f32), info=torch.empty((nl, L), dtype=torch.int32, device=dev),
             xsq2=torch.empty((L,), dtype=torch.float64, device=dev), alpha2=torch.empty((L,), **f32))
    lc.loca_error(z, cols, y, o["E"], ce=o["ce"])
    lc.loca_targets(o["E"], P, Q, o["T"], tsq=o["tsq"])
    lc.loca_gram_cross(X, o["T"], torch.ones((L,), **f32), o["gram"], o["cross"], zero_first=True)
    lc.loca_step_from_gram(o["gram"], o["tsq"], w.eta, o["xsq"], o["alpha"])
    lc.loca_ridge_solve(o["gram"], o["cross"], A, w.lambda_rel, o["B"], o["info"], xsq_total=o["xsq"],
                        cross_scale=o["alpha"])
    lc.loca_batch_step(X, o["tsq"], w.eta, o["xsq2"], o["alpha2"], zero_first=True)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    assert int(o["info"].abs().sum().item()) == 0
    return o


def _device_kspace(lc, w, inp, E):
    X, P, Q, A = (inp[k] for k in ("X", "P", "Q", "A"))
    L, d, C, k = w.L, w.d, w.C, w.k
    nl = len(w.lambda_rel)
    dev = X.device
    f32 = dict(dtype=torch.float32, device=dev)
    G = torch.empty((L, k, k), **f32)
    SC = torch.empty((L, C, k), **f32)
    xsq = torch.empty((L,), dtype=torch.float64, device=dev)
    B = torch.empty((nl, L, d, k), **f32)
    info = torch.empty((nl, L), dtype=torch.int32, device=dev)
    C_out = torch.empty((L, d, k), **f32)
    lc.loca_kspace_accumulate(X, A, E, P, Q, w.eta, G, SC, xsq, zero_first=True)
    lc.loca_kspace_solve(G, SC, P, Q, w.lambda_rel, B, info, xsq_total=xsq, C_out=C_out)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    assert int(info.abs().sum().item()) == 0
    return dict(G=G, C=C_out, B=B, xsq=xsq)


SINGLE = [
    # (workload, C override, also run the k-space path)
    ("qwen2.5-0.5b", 2, False),
    ("qwen2.5-0.5b", 3, False),
    ("qwen2.5-0.5b", 4, False),
    ("qwen2.5-7b", None, True),
    ("smollm2-1.7b", None, True),
    ("qwen2.5-14b", None, True),
]


@pytest.mark.parametrize("name,C,kspace", SINGLE, ids=[f"{n}-C{c}" if c else n for n, c, _ in SINGLE])
def test_single_batch_workload(lc, name, C, kspace):
    w = S.WORKLOADS[name]
    if C is not None:
        w = S.scaled(w, C=C, V=C)
    inp = S.device_inputs(w, seed=0, device="cuda")
    o = _device_chain(lc, w, inp)
    f = inp["host"]
    L, nl = w.L, len(w.lambda_rel)
    if w.V == w.C:
        E_ref, ce_ref = O.head_error(_np(inp["z"]), f["label_cols"], f["y"])
    else:
        E_ref, ce_ref = _oracle_error(inp["z"], inp["label_cols"], inp["y"])
    _check_error(o["E"], o["ce"], E_ref, ce_ref)
    del inp["z"]
    ks = _device_kspace(lc, w, inp, o["E"]) if kspace else None
    for l in (0, L - 1):
        X_h = _np(inp["X"][l])[None]
        ref = _oracle_block(E_ref, X_h, f, l, w, kspace=kspace)
        del X_h
        _check_targets(o["T"][l], ref["T"][0], E_ref, f["P"][l], f["Q"][l])
        assert abs(float(o["tsq"][l]) - ref["tsq"][0]) <= 1e-5 * ref["tsq"][0]
        x_ref = ref["xsq_total"][0]
        rx_trace = (float(o["xsq"][l]) - x_ref) / x_ref
        rx_sep = (float(o["xsq2"][l]) - x_ref) / x_ref
        print(f"{name} block {l}: ||X||^2 rel err, Gram trace {rx_trace:+.2e}, separate sum {rx_sep:+.2e}")
        assert abs(rx_sep) <= 2e-6
        # the tensor cores' fp32 accumulation drifts toward zero by a fraction of an ulp per MMA step;
        # restarting the accumulators every 16384 tokens bounds that drift to ~1e-4 of the sums
        assert abs(rx_trace) <= 1e-4
        assert abs(-float(o["alpha2"][l]) - ref["steps"][0]) <= 1e-5 * ref["steps"][0]
        cross_g = o["cross"][l] * o["alpha"][l]
        _check_stats(f"{name} block {l}", o["gram"][l], cross_g, o["B"][:, l], ref, nl)
        if ks is not None:
            rg = _rel(_np(ks["G"][l]), ref["Gk"][0])
            rc = _rel(_np(ks["C"][l]), ref["Ck"][0])
            rb = max(_rel(_np(ks["B"][j, l]), ref["Bk"][j, 0]) for j in range(nl))
            print(f"{name} block {l} k-space: rel err G {rg:.2e} C {rc:.2e} B {rb:.2e}")
            assert rg <= 2e-3 and rc <= 2e-3 and rb <= 2e-3
            assert abs(float(ks["xsq"][l]) - x_ref) <= 2e-6 * x_ref
        del ref
    del o, ks, inp
    _free()


# ----------------------------------------------------------------------------- streamed batches

def test_streamed_workload_qwen_1_5b(lc):
    """The 1.5B workload: 8 micro-batches of 8192 tokens, each through loca_targets and
    loca_accumulate (the step of that batch, then its Gram / cross contribution), the first with
    zero_first; then the solves.  The oracle streams the same batches (S7 additivity, one step per
    block and mini-batch, S8)."""
    from paper_2608_03020_gb300 import loca as lcm

    w = S.WORKLOADS["qwen2.5-1.5b"]
    assert w.micro_batches == 8 and w.tokens_per_batch == 8192
    inp = S.device_inputs(w, seed=0, device="cuda")
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    nb = w.tokens_per_batch
    batches = [X[:, n0:n0 + nb].contiguous() for n0 in range(0, w.N, nb)]
    ps = lcm.Pass(w.L, w.N, w.d, w.C, w.r, w.k, X.dtype, w.lambda_rel, w.eta, micro_batches=w.micro_batches)
    ps.run(z, cols, y, batches, P, Q, A)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    assert int(ps.info.abs().sum().item()) == 0
    f = inp["host"]
    E_ref, ce_ref = O.head_error(_np(z), f["label_cols"], f["y"])
    _check_error(ps.E, ps.ce, E_ref, ce_ref)
    nl = len(w.lambda_rel)
    for l in (0, w.L - 1):
        X_h = _np(X[l])[None]
        ref = _oracle_block(E_ref, X_h, f, l, w, micro_batches=w.micro_batches)
        del X_h
        # the Pass keeps the targets of the last micro-batch
        _check_targets(ps.T[l], ref["T"][0, w.N - nb:], E_ref[w.N - nb:], f["P"][l], f["Q"][l])
        x_ref = ref["xsq_total"][0]
        assert abs(float(ps.xsq[l]) - x_ref) <= 2e-6 * x_ref
        _check_stats(f"qwen2.5-1.5b block {l}", ps.gram[l], ps.cross[l], ps.B[:, l], ref, nl)
        del ref
    del ps, batches, inp, X
    _free()


# ----------------------------------------------------------------------------- scale reuse

def test_scale_reuse_smollm2(lc):
    """Prop. S8 with lambda_j = c_j tr(Gram_l)/d: scaling the adapter inputs X -> a X leaves every
    adapter of the candidate set unchanged.  For a = 4 (a power of two) every quantity of the chain
    scales exactly, so B agrees to rounding noise; for a = 3 the bf16 inputs round differently and
    B agrees within the bf16 tolerance.  Both the dense chain and the k-space path."""
    w = S.WORKLOADS["smollm2-1.7b"]
    inp = S.device_inputs(w, seed=0, device="cuda")
    X0 = inp["X"]
    o1 = _device_chain(lc, w, inp)
    k1 = _device_kspace(lc, w, inp, o1["E"])
    B1, Bk1 = o1["B"].clone(), k1["B"].clone()
    del o1, k1
    for a, tol in ((4.0, 1e-6), (3.0, 2e-3)):
        inp["X"] = (X0.float() * a).to(X0.dtype) if a != 4.0 else X0 * 4
        o2 = _device_chain(lc, w, inp)
        k2 = _device_kspace(lc, w, inp, o2["E"])
        rb = _rel(_np(o2["B"]), _np(B1))
        rk = _rel(_np(k2["B"]), _np(Bk1))
        print(f"scale {a}: B rel change dense {rb:.2e} (bitwise {torch.equal(o2['B'], B1)}), "
              f"k-space {rk:.2e} (bitwise {torch.equal(k2['B'], Bk1)})")
        assert rb <= tol and rk <= tol
        del o2, k2, inp["X"]
        _free()
    del inp, X0
    _free()
