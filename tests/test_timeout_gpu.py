"""The failure path of the bounded device waits, exercised without faulting or hanging the GPU.

A wait limit of 1 microsecond (the loca_set_wait_limit test hook) makes a wait of the
tensor-core kernels (targets, k-space statistics, the CTA-pair Gram / cross kernel with and
without generated targets, the ridge solve's projection) that has not succeeded after 8 polls
give up (a launch whose waits all succeed sooner finishes normally and must match the reference;
the test repeats the call until one gives up): the kernel must record
LOCA_ERR_TIMEOUT in the device status word, let its copies and MMAs in flight land, free its
tensor memory and return.  The CUDA context must stay usable: with the default limit restored,
the same call then gives results bit-identical to a call made before the failure, and the status
word reads OK.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

LOCA_ERR_TIMEOUT = 6


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    from paper_2608_03020_gb300 import loca

    loca.lib()
    yield loca
    loca.loca_set_wait_limit(0)


def _kspace_call(lc, X, A, E, P, Q):
    L, N, d = X.shape
    k, C = A.shape[2], E.shape[1]
    G = torch.empty((L, k, k), device="cuda")
    SC = torch.empty((L, C, k), device="cuda")
    xsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_kspace_accumulate(X, A, E, P, Q, 0.01, G, SC, xsq, zero_first=True)
    torch.cuda.synchronize()
    return G, SC, xsq


def _targets_call(lc, E, P, Q, L, N, d):
    T = torch.empty((L, N, d), dtype=torch.bfloat16, device="cuda")
    tsq = torch.empty((L,), dtype=torch.float64, device="cuda")
    lc.loca_targets(E, P, Q, T, tsq=tsq)
    torch.cuda.synchronize()
    return T, tsq


def _gram_call(lc, X, T):
    L, N, d = X.shape
    gram = torch.empty((L, d, d), device="cuda")
    cross = torch.empty((L, d, d), device="cuda")
    lc.loca_gram_cross(X, T, torch.full((L,), -0.5, device="cuda"), gram, cross, zero_first=True)
    torch.cuda.synchronize()
    return gram, cross


def _fused_call(lc, X, E, P, Q):
    L, N, d = X.shape
    gram = torch.empty((L, d, d), device="cuda")
    cross = torch.empty((L, d, d), device="cuda")
    lc.loca_gram_cross_fused(X, E, P, Q, torch.full((L,), 0.25, device="cuda"), gram, cross, zero_first=True)
    torch.cuda.synchronize()
    return gram, cross


def _ridge_call(lc, gram, cross, A):
    L, d, _ = gram.shape
    k = A.shape[2]
    B = torch.empty((2, L, d, k), device="cuda")
    info = torch.empty((2, L), dtype=torch.int32, device="cuda")
    lc.loca_ridge_solve(gram, cross, A, [1e-3, 1e-2], B, info)
    torch.cuda.synchronize()
    return B, info


def test_wait_timeout_is_reported_and_the_context_recovers(lc):
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    L, N, d, k, C, r = 4, 32768, 1024, 16, 4, 16
    X = torch.randn((L, N, d), device="cuda", generator=g).to(torch.bfloat16)
    A = torch.randn((L, d, k), device="cuda", generator=g) * 0.03
    E = torch.randn((N, C), device="cuda", generator=g)
    P = torch.randn((L, C, r), device="cuda", generator=g) * 0.25
    Q = torch.randn((L, r, d), device="cuda", generator=g) * 0.25
    lc.loca_set_wait_limit(0)
    assert lc.loca_device_status() == 0
    T = torch.randn((L, N, d), device="cuda", generator=g).to(torch.bfloat16)
    ref_k = _kspace_call(lc, X, A, E, P, Q)
    ref_t = _targets_call(lc, E, P, Q, L, N, d)
    ref_g = _gram_call(lc, X, T)
    ref_f = _fused_call(lc, X, E, P, Q)
    ref_r = _ridge_call(lc, ref_g[0], ref_g[1], A)
    assert lc.loca_device_status() == 0
    calls = {
        "kspace": lambda: _kspace_call(lc, X, A, E, P, Q),
        "targets": lambda: _targets_call(lc, E, P, Q, L, N, d),
        # the CTA-pair kernel: its roles stop at different points, the odd CTA's half of an armed
        # stage may never be issued, and every copy, MMA and bulk store still lands before either
        # CTA of a pair leaves
        "gram": lambda: _gram_call(lc, X, T),
        # the same kernel generating its targets: more roles (U producer, T conversion)
        "fused": lambda: _fused_call(lc, X, E, P, Q),
        # the tensor-core projection (d and k multiples of 4): producer, split groups, MMA and
        # epilogue rings
        "ridge": lambda: _ridge_call(lc, ref_g[0], ref_g[1], A),
    }
    refs = {"kspace": ref_k, "targets": ref_t, "gram": ref_g, "fused": ref_f, "ridge": ref_r}
    for call in calls:
        # 1 us: a wait that has not succeeded after 8 polls gives up.  A poll may suspend the
        # thread for a while, so a launch whose waits all complete within 8 polls finishes
        # normally; such a launch must then leave a clean status word and the reference results
        timed_out = False
        for attempt in range(10):
            lc.loca_set_wait_limit(1000)
            out = calls[call]()
            st = lc.loca_device_status()
            if st == LOCA_ERR_TIMEOUT:
                timed_out = True
                break
            assert st == 0, (call, attempt, st)
            lc.loca_set_wait_limit(0)
            for a, b in zip(refs[call], out):
                assert torch.equal(a, b), (call, attempt)
        assert timed_out, call
        lc.loca_set_wait_limit(0)
        again_k = _kspace_call(lc, X, A, E, P, Q)
        again_t = _targets_call(lc, E, P, Q, L, N, d)
        again_g = _gram_call(lc, X, T)
        again_f = _fused_call(lc, X, E, P, Q)
        again_r = _ridge_call(lc, ref_g[0], ref_g[1], A)
        assert lc.loca_device_status() == 0, call
        for a, b in zip(ref_k + ref_t + ref_g + ref_f + ref_r,
                        again_k + again_t + again_g + again_f + again_r):
            assert torch.equal(a, b), call
