"""Seeded synthetic inputs shaped like the paper's Qwen2.5 / SmolLM2 workloads.

This module draws random numbers and lays them out in the token-major layouts the
library takes.  It holds none of LoCA's arithmetic (no error, target, statistic or
solve); both the fp64 oracle and the CUDA path take their inputs from here and from
nowhere else.

Recipe (seed 0 unless stated):

* ``X_l[n, j] = g * s_{l,j}``, ``g ~ N(0, 1)``, per-channel scale ``s_{l,j} ~
  LogNormal(0, 0.5)`` drawn per block; from the 0.5B shape on, four seeded channels per
  block get a 20x scale (residual-stream outlier channels).  Stored as bf16 (round to
  nearest even) for the bf16 workloads, fp32 for the tiny one.
* Logits: when ``V == C`` (label-token head), ``z = X_L W_head`` with ``W_head ~
  N(0, 1/d)`` of shape ``d x C`` and ``X_L`` the last block's adapter input.  When
  ``V >> C`` (full vocabulary row), ``z ~ N(0, 1)`` i.i.d. plus an offset of
  ``log(V / C)`` on the ``C`` label columns so that they hold about half of the softmax
  mass; stored as bf16.
* Labels ``y ~ U{0..C-1}``; label columns are ``0..C-1`` when ``V == C`` and ``C``
  distinct seeded positions otherwise.
* Feedback factors ``P_l ~ N(0, 1/r)`` (``C x r``), ``Q_l ~ N(0, 1/r)`` (``r x d``).
* Fixed down-projection ``A_l``: QR of a Gaussian ``d x k`` with ``diag(R) > 0``
  (orthonormal columns).
* Probe pairs for the calibration fit: ``E_probe ~ N(0, 1)`` (``Np x m``) and
  ``G_probe_l = E_probe M_l + 0.1 * rms(E_probe M_l) * noise`` with ``M_l`` a planted
  rank-``min(rank, m)`` map.  For the paper's d-wide error space (``m = d``) the columns
  of ``E_probe`` optionally get LogNormal(0, 0.5) scales, so that ``E^T E`` is
  anisotropic like an unembedded error (``e_scales=True``).
* Test matrix of the randomized top-r fit: ``Omega ~ N(0, 1)`` (``d x ell``).

Host generation (numpy) serves the small shapes the oracle runs in full; device
generation (torch on CUDA) serves the full-size shapes, whose small factors
(``P, Q, A, y, label_cols, W_head``, channel scales) are still drawn on the host with
numpy so that both sides see identical values.
"""

from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass

import numpy as np

# tensor ids used to derive independent streams from one seed
_S_SCALE, _S_X, _S_HEAD, _S_Y, _S_COLS, _S_P, _S_Q, _S_A, _S_Z, _S_PE, _S_PM, _S_PN, _S_OUT, _S_BPREV, _S_OMEGA, _S_PSC = range(1, 17)


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: shapes, dtypes and hyper-parameters."""

    name: str
    L: int  # transformer blocks
    d: int  # hidden width
    N: int  # tokens per pass
    C: int  # label classes (columns of E)
    V: int  # logit row width (== C for a label-token head)
    r: int  # feedback rank (columns of P, rows of Q)
    k: int  # adapter rank (columns of A and B)
    act_dtype: str = "bf16"  # X and the GEMM feed of T: "bf16" or "f32"
    logit_dtype: str = "f32"
    lambda_rel: tuple = (1e-4, 1e-3, 1e-2)
    eta: float = 0.01
    micro_batches: int = 1
    outliers: int = 4
    seqs: int = 0  # sequences x 256 tokens (informational)

    @property
    def tokens_per_batch(self) -> int:
        return -(-self.N // self.micro_batches)


WORKLOADS = {
    "tiny": Workload("tiny", L=2, d=64, N=512, C=4, V=4, r=4, k=4, act_dtype="f32",
                     lambda_rel=(1e-2,), outliers=0),
    "qwen2.5-0.5b": Workload("qwen2.5-0.5b", L=24, d=896, N=16384, C=4, V=4, r=8, k=8, seqs=64),
    "qwen2.5-1.5b": Workload("qwen2.5-1.5b", L=28, d=1536, N=65536, C=4, V=4, r=16, k=16,
                             micro_batches=8, seqs=256),
    "qwen2.5-7b": Workload("qwen2.5-7b", L=28, d=3584, N=131072, C=4, V=4, r=16, k=16, seqs=512),
    "qwen2.5-14b": Workload("qwen2.5-14b", L=48, d=5120, N=131072, C=4, V=151936, r=32, k=32,
                            logit_dtype="bf16", seqs=512),
    "smollm2-1.7b": Workload("smollm2-1.7b", L=24, d=2048, N=131072, C=4, V=49152, r=32, k=32,
                             logit_dtype="bf16", seqs=512),
}


def scaled(w: Workload, **changes) -> Workload:
    """A copy of ``w`` with some fields changed (smaller L or N for parity runs)."""
    return dataclasses.replace(w, **changes)


def _rng(seed: int, *ids: int) -> np.random.Generator:
    return np.random.default_rng(np.random.SeedSequence([int(seed), *[int(i) for i in ids]]))


def _to_bf16_values(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest even) and return them as fp32."""
    import torch

    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    return t.to(torch.bfloat16).to(torch.float32).numpy()


def channel_scales(w: Workload, seed: int, l: int) -> np.ndarray:
    """Per-channel scales ``s_{l,j}`` of block ``l`` (LogNormal(0, 0.5), outliers x20)."""
    s = _rng(seed, _S_SCALE, l).lognormal(0.0, 0.5, size=w.d)
    if w.outliers:
        idx = _rng(seed, _S_OUT, l).choice(w.d, size=min(w.outliers, w.d), replace=False)
        s[idx] *= 20.0
    return s


def host_factors(w: Workload, seed: int = 0) -> dict:
    """The small inputs (everything except X and full-vocabulary logits) as numpy arrays."""
    L, d, N, C, V, r, k = w.L, w.d, w.N, w.C, w.V, w.r, w.k
    y = _rng(seed, _S_Y).integers(0, C, size=N).astype(np.int32)
    if V == C:
        cols = np.arange(C, dtype=np.int32)
    else:
        cols = np.sort(_rng(seed, _S_COLS).choice(V, size=C, replace=False)).astype(np.int32)
    P = np.stack([_rng(seed, _S_P, l).normal(0.0, 1.0 / math.sqrt(r), size=(C, r)) for l in range(L)])
    Q = np.stack([_rng(seed, _S_Q, l).normal(0.0, 1.0 / math.sqrt(r), size=(r, d)) for l in range(L)])
    A = np.empty((L, d, k))
    for l in range(L):
        g = _rng(seed, _S_A, l).normal(size=(d, k))
        q, rr = np.linalg.qr(g)
        A[l] = q * np.sign(np.diag(rr))[None, :]
    W_head = _rng(seed, _S_HEAD).normal(0.0, 1.0 / math.sqrt(d), size=(d, C)) if V == C else None
    s = np.stack([channel_scales(w, seed, l) for l in range(L)])
    return dict(y=y, label_cols=cols, P=P.astype(np.float32), Q=Q.astype(np.float32),
                A=A.astype(np.float32), W_head=None if W_head is None else W_head.astype(np.float32),
                scales=s, lambda_rel=np.asarray(w.lambda_rel, dtype=np.float32), eta=np.float32(w.eta))


def host_B_prev(w: Workload, seed: int = 0, scale: float = 0.01) -> np.ndarray:
    """A nonzero current adapter ``B^(t)`` (``L x d x k``) for second-iteration runs."""
    return (scale * _rng(seed, _S_BPREV).normal(size=(w.L, w.d, w.k))).astype(np.float32)


def host_X(w: Workload, seed: int = 0) -> np.ndarray:
    """Adapter inputs ``X`` (``L x N x d``) drawn on the host; bf16 values for bf16 workloads."""
    f = host_factors(w, seed)
    X = np.empty((w.L, w.N, w.d), dtype=np.float32)
    for l in range(w.L):
        X[l] = _rng(seed, _S_X, l).standard_normal(size=(w.N, w.d)) * f["scales"][l][None, :]
    if w.act_dtype == "bf16":
        X = _to_bf16_values(X)
    return X


def host_logits(w: Workload, X: np.ndarray | None, seed: int = 0) -> np.ndarray:
    """Logits ``N x V`` (fp32 values; bf16-representable when ``logit_dtype == 'bf16'``)."""
    f = host_factors(w, seed)
    if w.V == w.C:
        z = (X[w.L - 1].astype(np.float64) @ f["W_head"].astype(np.float64)).astype(np.float32)
    else:
        z = _rng(seed, _S_Z).standard_normal(size=(w.N, w.V)).astype(np.float32)
        z[:, f["label_cols"]] += np.float32(math.log(w.V / w.C))
    if w.logit_dtype == "bf16":
        z = _to_bf16_values(z)
    return z


def host_inputs(w: Workload, seed: int = 0) -> dict:
    """Every input of one pass as numpy arrays (small shapes only)."""
    f = host_factors(w, seed)
    X = host_X(w, seed)
    f["X"] = X
    f["z"] = host_logits(w, X, seed)
    return f


def probe_error_scales(m: int, seed: int = 0) -> np.ndarray:
    """Column scales of ``E_probe`` for ``e_scales=True`` (LogNormal(0, 0.5), ``m``)."""
    return _rng(seed, _S_PSC).lognormal(0.0, 0.5, size=m)


def planted_factors(m: int, d: int, rank: int, seed: int, l: int) -> tuple[np.ndarray, np.ndarray]:
    """The two factors of block ``l``'s planted map ``M_l = a b / sqrt(rho)``, ``rho = min(rank, m)``."""
    rho = min(rank, m)
    g = _rng(seed, _S_PM, l)
    return g.standard_normal(size=(m, rho)), g.standard_normal(size=(rho, d))


def host_probe_pairs(Np: int, m: int, d: int, L: int, rank: int, noise: float = 0.1,
                     seed: int = 0, e_scales: bool = False) -> dict:
    """Probe pairs for the calibration fit: ``E_probe`` (``Np x m``), ``G_probe`` (``L x Np x d``),
    and the planted maps ``M`` (``L x m x d``, rank ``min(rank, m)``)."""
    E = _rng(seed, _S_PE).standard_normal(size=(Np, m))
    if e_scales:
        E = E * probe_error_scales(m, seed)[None, :]
    rho = min(rank, m)
    M = np.empty((L, m, d))
    G = np.empty((L, Np, d))
    for l in range(L):
        a, b = planted_factors(m, d, rank, seed, l)
        M[l] = (a @ b) / math.sqrt(rho)
        clean = E @ M[l]
        nz = _rng(seed, _S_PN, l).standard_normal(size=(Np, d))
        G[l] = clean + noise * math.sqrt(float(np.mean(clean ** 2))) * nz
    return dict(E_probe=E.astype(np.float32), G_probe=G.astype(np.float32), M=M)


def device_probe_pairs(Np: int, m: int, d: int, L: int, rank: int, noise: float = 0.1, seed: int = 0,
                       e_scales: bool = True, device="cuda") -> dict:
    """Full-size probe pairs drawn on ``device`` with the recipe of :func:`host_probe_pairs`
    (seeded CUDA generator for the ``Np``-row arrays; the planted factors and column scales
    from the host streams).  Returns fp32 ``E_probe`` (``Np x m``) and ``G_probe``
    (``L x Np x d``)."""
    import torch

    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) * 1_000_003 + _S_PE)
    E = torch.randn((Np, m), generator=gen, device=device, dtype=torch.float32)
    if e_scales:
        E *= torch.from_numpy(probe_error_scales(m, seed).astype(np.float32)).to(device)[None, :]
    rho = min(rank, m)
    G = torch.empty((L, Np, d), device=device, dtype=torch.float32)
    for l in range(L):
        a, b = planted_factors(m, d, rank, seed, l)
        Ml = torch.from_numpy(((a @ b) / math.sqrt(rho)).astype(np.float32)).to(device)
        clean = E @ Ml
        gen.manual_seed(int(seed) * 1_000_003 + 7919 * (l + 1) + _S_PN)
        nz = torch.randn((Np, d), generator=gen, device=device, dtype=torch.float32)
        G[l] = clean + noise * torch.sqrt(torch.mean(clean * clean)) * nz
        del Ml, clean, nz
    return dict(E_probe=E, G_probe=G)


def omega_matrix(d: int, ell: int, seed: int = 0) -> np.ndarray:
    """Gaussian test matrix ``Omega`` (``d x ell``, fp32) of the randomized top-r fit."""
    return _rng(seed, _S_OMEGA).standard_normal(size=(d, ell)).astype(np.float32)


def device_inputs(w: Workload, seed: int = 0, device="cuda", x_source: str = "device",
                  with_logits: bool = True) -> dict:
    """Every input of one pass as torch tensors on ``device``.

    ``x_source="host"`` copies :func:`host_X` (small shapes, so the oracle sees the same
    values); ``"device"`` draws ``X`` block by block with a seeded CUDA generator.
    """
    import torch

    f = host_factors(w, seed)
    out = {}
    act = torch.bfloat16 if w.act_dtype == "bf16" else torch.float32
    if x_source == "host":
        X = torch.from_numpy(host_X(w, seed)).to(device=device, dtype=act)
    else:
        X = torch.empty((w.L, w.N, w.d), dtype=act, device=device)
        gen = torch.Generator(device=device)
        for l in range(w.L):
            gen.manual_seed(int(seed) * 1_000_003 + 7919 * (l + 1) + _S_X)
            s = torch.from_numpy(f["scales"][l].astype(np.float32)).to(device)
            for n0 in range(0, w.N, 32768):
                n1 = min(w.N, n0 + 32768)
                g = torch.randn((n1 - n0, w.d), generator=gen, device=device, dtype=torch.float32)
                X[l, n0:n1] = (g * s[None, :]).to(act)
    out["X"] = X
    if with_logits:
        if w.V == w.C:
            Wh = torch.from_numpy(f["W_head"]).to(device)
            z = X[w.L - 1].float() @ Wh
        else:
            gen = torch.Generator(device=device)
            gen.manual_seed(int(seed) * 1_000_003 + _S_Z)
            ldt = torch.bfloat16 if w.logit_dtype == "bf16" else torch.float32
            z = torch.empty((w.N, w.V), dtype=ldt, device=device)
            cols = torch.from_numpy(f["label_cols"].astype(np.int64)).to(device)
            off = float(math.log(w.V / w.C))
            for n0 in range(0, w.N, 8192):
                n1 = min(w.N, n0 + 8192)
                g = torch.randn((n1 - n0, w.V), generator=gen, device=device, dtype=torch.float32)
                g[:, cols] += off
                z[n0:n1] = g.to(ldt)
        if w.logit_dtype == "bf16":
            z = z.to(torch.bfloat16)
        out["z"] = z.contiguous()
    for key in ("y", "label_cols"):
        out[key] = torch.from_numpy(f[key]).to(device)
    for key in ("P", "Q", "A"):
        out[key] = torch.from_numpy(f[key]).to(device)
    out["host"] = f
    return out
