"""Full-size parity at the Qwen2.5-7B statistics shape (L = 28, N = 131072, d = 3584, C = 4,
r = k = 16), in the launch configuration ``bench.py`` times: the same seeded inputs, the same
sequence of C-ABI calls over all 28 blocks at once (error, targets, Gram / cross at alpha = 1,
the step from the Gram trace, the solve with alpha as cross_scale).  The separate step
(``loca_batch_step``) runs on the same inputs too.  The fp64 oracle then recomputes the whole
chain (head error, targets, step, Gram / cross, projection, ridge solves) for two of the blocks
(the first and the last) over all N tokens, and every output of those blocks is compared
element by element.  The tolerances are the parity tests' own (see ``test_parity_gpu``).
"""

import numpy as np
import pytest
import torch

from oracle import loca_oracle as O
from synth import inputs as S

pytestmark = pytest.mark.gpu


def _np(t):
    return t.detach().float().cpu().numpy().astype(np.float64) if t.dtype != torch.float64 else t.cpu().numpy()


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a) - np.asarray(b)) / max(np.linalg.norm(np.asarray(b)), 1e-300))


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    from paper_2608_03020_gb300 import loca

    loca.lib()
    return loca


def test_qwen7b_shape_full_pass_two_blocks(lc):
    w = S.WORKLOADS["qwen2.5-7b"]
    inp = S.device_inputs(w, seed=0, device="cuda")
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, r, k = w.L, w.N, w.d, w.C, w.r, w.k
    nl = len(w.lambda_rel)
    dev = X.device
    f32 = dict(dtype=torch.float32, device=dev)
    E = torch.empty((N, C), **f32)
    ce = torch.empty((N,), **f32)
    T = torch.empty((L, N, d), dtype=X.dtype, device=dev)
    tsq = torch.empty((L,), dtype=torch.float64, device=dev)
    xsq = torch.empty((L,), dtype=torch.float64, device=dev)
    alpha = torch.empty((L,), **f32)
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    B = torch.empty((nl, L, d, k), **f32)
    info = torch.empty((nl, L), dtype=torch.int32, device=dev)
    xsq2 = torch.empty((L,), dtype=torch.float64, device=dev)
    alpha2 = torch.empty((L,), **f32)
    lc.loca_error(z, cols, y, E, ce=ce)
    lc.loca_targets(E, P, Q, T, tsq=tsq)
    lc.loca_gram_cross(X, T, torch.ones((L,), **f32), gram, cross, zero_first=True)
    lc.loca_step_from_gram(gram, tsq, w.eta, xsq, alpha)
    lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, cross_scale=alpha)
    lc.loca_batch_step(X, tsq, w.eta, xsq2, alpha2, zero_first=True)
    torch.cuda.synchronize()
    assert lc.loca_device_status() == 0
    assert int(info.abs().sum().item()) == 0

    h = inp["host"]
    z_h = _np(z)
    E_g = _np(E)
    for l in (0, L - 1):
        X_h = X[l].float().cpu().numpy()[None].astype(np.float64)
        ref = O.loca_pass(z_h, h["label_cols"], h["y"], X_h, h["P"][l:l + 1], h["Q"][l:l + 1],
                          h["A"][l:l + 1], w.eta, w.lambda_rel, t_feed="bf16")
        if l == 0:
            # head error, all tokens: fp32 softmax of 4 logits -> 1e-5 of the loss weight (1)
            assert np.max(np.abs(E_g - ref["E"])) <= 1e-5
        # targets: within half a bf16 ulp, plus the fp32 bound of the products (relative to the
        # magnitude sum (|E| |P|) |Q| of all terms), plus the GPU head error's own absolute error
        # carried through P Q: for the true label E = p - 1 is formed in fp32, so near p = 1 it
        # has an absolute error of up to ~6e-8 whatever its size (1e-6 allowed, 16x margin)
        T_g = _np(T[l])
        T_r = ref["T"][0]
        Pa = np.abs(h["P"][l].astype(np.float64))
        Qa = np.abs(h["Q"][l].astype(np.float64))
        scale = (np.abs(ref["E"]) @ Pa) @ Qa
        e_abs = (np.ones((1, C)) @ Pa) @ Qa
        _, e = np.frexp(T_r)
        bound = 1e-5 * scale + 1e-6 * e_abs + np.ldexp(1.0, e - 9) + 1e-30
        assert np.all(np.abs(T_g - T_r) <= bound), (l, float(np.max(np.abs(T_g - T_r) - bound)))
        del T_g, T_r, scale, e, bound
        assert abs(float(tsq[l]) - ref["tsq"][0]) <= 1e-5 * ref["tsq"][0]
        # ||X_l||^2 from the separate step (exact squares, fp32 partials of 32 terms summed in
        # fp64) and from the Gram trace: each diagonal entry is the tensor cores' fp32
        # accumulation of 131072 products, which carries ~1e-3 relative (measured 6.5e-4), so the
        # step alpha = -eta sqrt(xsq / tsq) agrees with the separate step to half that
        x_ref = ref["xsq_total"][0]
        print(f"block {l}: xsq rel err, Gram trace {(float(xsq[l]) - x_ref) / x_ref:+.2e}, "
              f"separate step {(float(xsq2[l]) - x_ref) / x_ref:+.2e}")
        assert abs(float(xsq2[l]) - x_ref) <= 2e-6 * x_ref
        assert abs(float(xsq[l]) - x_ref) <= 1e-3 * x_ref
        assert abs(float(alpha[l]) - float(alpha2[l])) <= 5e-4 * abs(float(alpha2[l]))
        gg, cg = _np(gram[l]), _np(cross[l]) * float(alpha[l])
        assert np.array_equal(gg, gg.T)
        rg, rc = _rel(gg, ref["gram"][0]), _rel(cg, ref["cross"][0])
        print(f"block {l}: rel err gram {rg:.2e} cross {rc:.2e}")
        assert rg <= 2e-3 and rc <= 2e-3
        for j in range(nl):
            rb = _rel(_np(B[j, l]), ref["B"][j, 0])
            print(f"block {l} lambda {j}: rel err B {rb:.2e}")
            assert rb <= 2e-3
        del ref, X_h
