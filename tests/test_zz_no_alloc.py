"""loca_accumulate_noalloc: the statistics entry point for callers that cannot allocate device
memory when they call the library (its scratch is a fixed array inside the library).

Checks, through the C ABI on the GPU, that two calls in a row (the second accumulating onto
the first) give the same statistics as loca_accumulate with a caller workspace, within the
tolerances the other statistics tests use (2e-3 relative Frobenius for bf16 inputs, 1e-5 for
fp32 inputs; both paths are deterministic, so the results are in fact identical), and that a
block count above the array's limit is refused.  Collected last so that a run which stops at
the first failure has already run every other test; it also passes alone in a fresh process.
"""

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lc():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_03020_gb300 import _build

    _build.build()
    from paper_2608_03020_gb300 import loca

    loca.lib()
    return loca


def _inputs(L, N, d, dtype, seed):
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    scale = torch.exp(0.5 * torch.randn((L, 1, d), generator=g, device="cuda"))
    X = (torch.randn((L, N, d), generator=g, device="cuda") * scale).to(dtype)
    T = (0.05 * torch.randn((L, N, d), generator=g, device="cuda")).to(dtype)
    tsq = (T.double() ** 2).sum(dim=(1, 2))
    return X, T, tsq


def _rel(a, b):
    return float(torch.linalg.norm((a - b).double()) / torch.linalg.norm(b.double()))


@pytest.mark.parametrize("dtype,L,N,d,tol", [
    (torch.bfloat16, 3, 1000, 328, 2e-3),
    (torch.float32, 2, 300, 72, 1e-5),
])
def test_noalloc_matches_workspace_entry_point_on_two_calls(lc, dtype, L, N, d, tol):
    batches = [_inputs(L, N, d, dtype, 1), _inputs(L, N // 2 + 3, d, dtype, 2)]
    outs = []
    for use_noalloc in (False, True):
        gram = torch.full((L, d, d), float("nan"), device="cuda")
        cross = torch.full((L, d, d), float("nan"), device="cuda")
        xsq = torch.full((L,), float("nan"), dtype=torch.float64, device="cuda")
        for i, (X, T, tsq) in enumerate(batches):
            if use_noalloc:
                lc.loca_accumulate_noalloc(X, T, tsq, 0.01, gram, cross, xsq, zero_first=(i == 0))
            else:
                lc.loca_accumulate(X, T, tsq, 0.01, gram, cross, xsq, zero_first=(i == 0))
        torch.cuda.synchronize()
        outs.append((gram, cross, xsq))
    assert lc.loca_device_status() == 0
    (g0, c0, x0), (g1, c1, x1) = outs
    assert _rel(g1, g0) <= tol and _rel(c1, c0) <= tol
    assert torch.allclose(x1, x0, rtol=1e-12, atol=0)
    assert torch.equal(g1, g0) and torch.equal(c1, c0) and torch.equal(x1, x0)


def test_noalloc_rejects_more_blocks_than_its_scratch_holds(lc):
    L, N, d = 65, 8, 8
    X = torch.zeros((L, N, d), dtype=torch.bfloat16, device="cuda")
    tsq = torch.zeros((L,), dtype=torch.float64, device="cuda")
    gram = torch.zeros((L, d, d), device="cuda")
    xsq = torch.zeros((L,), dtype=torch.float64, device="cuda")
    with pytest.raises(lc.LocaError) as exc:
        lc.loca_accumulate_noalloc(X, X, tsq, 0.01, gram, gram.clone(), xsq, zero_first=True)
    assert exc.value.status == 2
    assert "L <= 64" in str(exc.value)
