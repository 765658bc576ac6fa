#!/usr/bin/env python3
"""Throughput of one LoCA Stage-II pass on GB300: tokens/s/block at the Qwen2.5-7B shape.

A step is one pass of the whole hot path over one batch of synthetic inputs resident in HBM:
  loca_error -> loca_targets -> loca_gram_cross -> loca_step_from_gram -> loca_ridge_solve
(head error, feedback targets, Gram / cross statistics on the tensor cores, the
scale-normalised step from tr(Gram) = ||X||^2 of the one mini-batch, projected ridge solves for
every block and every candidate lambda with the step applied to the cross product).

value     = N * L / (seconds per step)            tokens per second per block (higher is better)
e2e       = the same metric with the inputs copied from pinned host memory and the adapters
            copied back inside every timed step; X (26 GB) streams in through
            loca_accumulate_streamed, its copies overlapping the statistics kernels
roofline  = the Gram / cross kernel (the dominant one): useful flops per launch
            L * (2 N d^2 + N d (d + 1)) over its CUDA-event duration, against the measured
            sustained bf16 peak
cpu_baseline = the fp64 oracle on the host cores on a bounded sample (one block, a prefix of
            the tokens)

Inputs (X is 26 GB at 7B) are far larger than the 129 MB L2, so no flush is needed between
steps.  --impl reference times the oracle itself (the reference arm of this comparison).
Multi-GPU: the method needs one GPU; --gpus N runs N independent replicas (weak scaling),
with a barrier and the max step time over ranks.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "LoCA fit tokens/s/block at Qwen2.5-7B shape, 1 GB300; % bf16 tensor-core peak"
UNIT = "tokens/s/block"
FALLBACK_SUSTAINED_TFLOPS = 1700.0  # profiling recipe's sustained figure, used if no measured file

# DRAM bytes (read + write) per launch from an ncu capture of a small case of the same kernel
# (L_capture blocks at the workload's own N and d: a few GB on the device), valid only for the
# kernel source whose sha256 prefix is given.  Work items and rounds repeat block by block, so
# the traffic of a launch over L blocks is the capture's times L / L_capture; any other N, d or
# k, or another source, reports null.
GRAM_TC_TRAFFIC = {"sha256": "81575fe3750817bb", "L_capture": 2, "N": 131072, "d": 3584,
                   "read": 8478698496, "write": 1255207936,
                   "kernel": "k_gram_cross_tc"}
# k_kspace_xa (the k-space statistics kernel, which reads X) at k = 16
KSPACE_TRAFFIC = {"sha256": "3aba9c60b10e48c0", "L_capture": 2, "N": 131072, "d": 3584, "k": 16,
                  "read": 1885266176, "write": 2223872,
                  "kernel": "k_kspace_xa"}
# k_targets_tc (writes T) at r = 16, bf16 output
TARGETS_TRAFFIC = {"sha256": "1796bbc513a2c2d2", "L_capture": 2, "N": 131072, "d": 3584, "r": 16,
                   "read": 13250816, "write": 1817000448,
                   "kernel": "k_targets_tc"}
# k_project_tc (the ridge solve's projection, which reads Gram and Cross once) at k = 16: taken
# on the full launch (L = 28, 2.9 GB of statistics), so L_capture = 28
PROJECT_TRAFFIC = {"sha256": "7771065c47a83799", "L_capture": 28, "d": 3584, "k": 16,
                   "read": 2886107648, "write": 17300992,
                   "kernel": "k_project_tc"}


def recorded_traffic(rec, source_file, L, **shape):
    """DRAM bytes per launch over L blocks from a small-case capture record, or None once the
    kernel source or the shape (every key of ``shape``, which the record must hold) differs."""
    src = open(os.path.join(ROOT, "paper_2608_03020_gb300", "csrc", source_file), "rb").read()
    if rec["sha256"] != hashlib.sha256(src).hexdigest()[:16] or any(rec[n] != v for n, v in shape.items()):
        return None
    return float(rec["read"] + rec["write"]) * L / rec["L_capture"]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default="qwen2.5-7b")
    ap.add_argument("--L", type=int, default=None, help="override the workload's block count")
    ap.add_argument("--N", type=int, default=None, help="override the workload's token count")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-kspace", action="store_true", help="skip the k-space statistics measurement")
    ap.add_argument("--no-vocab", action="store_true", help="skip the wide-vocabulary head-error measurement")
    ap.add_argument("--vocab-N", type=int, default=None,
                    help="token count of the wide-vocabulary head-error leg (default: the 14B workload's 131072)")
    ap.add_argument("--no-calib", action="store_true", help="skip the one-shot d-wide feedback-fit measurement")
    ap.add_argument("--e2e-group", type=int, default=2, help="blocks per host-to-device copy in the e2e leg")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the other workloads' own-shape measurements")
    ap.add_argument("--no-fused", action="store_true", help="skip the fused-targets pass")
    ap.add_argument("--ridge-only", action="store_true",
                    help="time loca_ridge_solve alone on seeded statistics of the workload's shape (for profiling)")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            mp = json.load(f)
        return float(mp["bf16_tflops_sustained"]), "measured"
    return FALLBACK_SUSTAINED_TFLOPS, "fallback"


def hbm_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            return float(json.load(f)["hbm_gbs"])
    return 6800.0  # the profiling recipe's fallback copy rate


class ClockSampler:
    """nvidia-smi samples (200 ms) of SM and memory clocks, power and throttle reasons during the
    timed region (read only)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap,"
              "clocks.mem,clocks.max.mem")

    def __init__(self, uuid):
        self.uuid = uuid
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            args = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
            if self.uuid:
                args += ["-i", self.uuid]
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(args, stdout=self.out, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.out.close()

    def summary(self):
        if self.proc is None or self.path is None:
            return None
        rows, extra = [], []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
            try:
                extra.append((float(parts[3]), float(parts[9]), float(parts[10])))
            except (ValueError, IndexError):
                pass
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows for i, v in enumerate(flags) if v.lower() == "active"})
        out = {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
               "reasons": reasons, "samples": len(rows)}
        if extra:
            out.update({"power_w": statistics.median(e[0] for e in extra),
                        "mem_mhz": statistics.median(e[1] for e in extra), "mem_max_mhz": max(e[2] for e in extra)})
        return out


def dist_setup(args):
    import torch

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def max_over_ranks(world, value):
    if world == 1:
        return value
    import torch
    import torch.distributed as dist

    t = torch.tensor([value], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- oracle timing

def oracle_sample(w, tokens, host):
    """One oracle pass on a bounded sample: block 0, the first `tokens` tokens."""
    import numpy as np

    from oracle import loca_oracle as O

    X = host["X0"][:tokens][None].astype(np.float64)
    t0 = time.perf_counter()
    O.loca_pass(host["z"][:tokens], host["label_cols"], host["y"][:tokens], X, host["P"][:1], host["Q"][:1],
                host["A"][:1], w.eta, w.lambda_rel, t_feed="bf16" if w.act_dtype == "bf16" else None)
    return time.perf_counter() - t0


def host_sample(w, seed=0, tokens=None):
    """Host-side inputs for the oracle sample (block 0 drawn with the same recipe)."""
    import numpy as np

    from synth import inputs as S

    f = S.host_factors(w, seed)
    n = tokens or w.N
    ws = S.scaled(w, L=1, N=n)
    X0 = S.host_X(ws, seed)[0]
    if w.V == w.C:
        z = (X0.astype(np.float64) @ f["W_head"].astype(np.float64)).astype(np.float32)
    else:
        z = S.host_logits(S.scaled(w, N=n), None, seed)
    return dict(X0=X0, z=z, y=f["y"][:n], label_cols=f["label_cols"], P=f["P"], Q=f["Q"], A=f["A"])


def run_reference(args, w):
    tokens = min(2048, w.N)  # bounded sample per step, capped at the workload's N
    host = host_sample(w, tokens=tokens)
    for _ in range(args.warmup):
        oracle_sample(w, tokens, host)
    times = [oracle_sample(w, tokens, host) for _ in range(args.steps)]
    sec = sum(times) / len(times)
    value = tokens / sec
    cores = os.cpu_count()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "L": w.L, "d": w.d, "N": w.N, "C": w.C, "r": w.r, "k": w.k,
                   "sample": f"block 0, first {tokens} tokens"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"one block (of {w.L}), first {tokens} of {w.N} tokens, full d={w.d}; numpy fp64"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# ----------------------------------------------------------------------------- host description

def host_cpu():
    """Host CPU as lscpu reports it (model, logical CPUs) and the oracle's BLAS thread count."""
    out = {"cores": os.cpu_count()}
    try:
        txt = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=20).stdout
        for line in txt.splitlines():
            k, _, v = line.partition(":")
            k, v = k.strip(), v.strip()
            if k in ("Architecture", "Model name", "CPU(s)", "Thread(s) per core", "Core(s) per socket", "Socket(s)"):
                out[k.lower().replace("(s)", "s").replace(" ", "_")] = v
    except Exception as e:  # lscpu missing: report what Python sees
        out["lscpu"] = f"unavailable: {e}"
    return out


def tiny_oracle_times():
    """The fp64 oracle's full pass on the tiny workload (every block and token), with BLAS on all
    host cores (this process) and single-threaded (a fresh interpreter with one BLAS thread)."""
    code = ("import time, sys; sys.path.insert(0, %r); from synth import inputs as S; from oracle import loca_oracle as O; "
            "w = S.WORKLOADS['tiny']; f = S.host_inputs(w); "
            "run = lambda: O.loca_pass(f['z'], f['label_cols'], f['y'], f['X'], f['P'], f['Q'], f['A'], w.eta, w.lambda_rel); "
            "run(); t = time.perf_counter(); [run() for _ in range(5)]; print((time.perf_counter() - t) / 5)") % ROOT
    res = {}
    for name, threads in (("all_cores_s", None), ("single_thread_s", "1")):
        env = dict(os.environ)
        if threads:
            for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
                env[v] = threads
        try:
            r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=300)
            res[name] = float(r.stdout.strip().splitlines()[-1])
        except Exception as e:
            res[name] = f"failed: {e}"
    return res


# ----------------------------------------------------------------------------- other workloads

def write_peak(buf, stream, reps=3):
    """Write-only HBM rate of this GPU in this run: torch's fill of ``buf`` (larger than L2)."""
    import torch

    buf.zero_()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(reps):
        buf.zero_()
    b.record(stream)
    torch.cuda.synchronize()
    return reps * buf.numel() * buf.element_size() / (a.elapsed_time(b) / 1e3) / 1e9


def hbm_object(nbytes, ms, kernel, hbm, wpeak=None):
    gbs = nbytes / (ms / 1e3) / 1e9
    o = {"bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s", "frac": gbs / hbm, "kernel": kernel,
         "bytes_per_launch": float(nbytes), "ms": ms}
    if wpeak:
        o["write_peak_gbs"] = wpeak
        o["frac_of_write_peak"] = gbs / wpeak
    return o


def measure_workload(lc, name, dev, stream, steps, warmup, peak, hbm, wpeak):
    """One step of workload `name` at its own shape, timed like the headline: error -> targets ->
    statistics -> solve (single mini-batch: the cross product at alpha = 1, the step from the Gram
    trace, alpha in the solve; several mini-batches: targets and loca_accumulate per batch)."""
    import torch

    from synth import inputs as S

    w = S.WORKLOADS[name]
    inp = S.device_inputs(w, seed=0, device=dev)
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, r, k = w.L, w.N, w.d, w.C, w.r, w.k
    mb, nb = w.micro_batches, w.tokens_per_batch
    nl = len(w.lambda_rel)
    act = X.dtype
    if mb > 1:  # contiguous per-batch inputs (L x nb x d each)
        X = X.view(L, mb, nb, d).permute(1, 0, 2, 3).contiguous()
        inp["X"] = None
    f32 = dict(dtype=torch.float32, device=dev)
    E = torch.empty((N, C), **f32)
    ce = torch.empty((N,), **f32)
    T = torch.empty((L, nb, d), dtype=act, device=dev)
    tsq = torch.empty((L,), dtype=torch.float64, device=dev)
    xsq = torch.empty((L,), dtype=torch.float64, device=dev)
    alpha = torch.empty((L,), **f32)
    ones = torch.ones((L,), **f32)
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    B = torch.empty((nl, L, d, k), **f32)
    info = torch.empty((nl, L), dtype=torch.int32, device=dev)
    ws_t = torch.empty(lc.targets_workspace_size(nb, L, d), dtype=torch.uint8, device=dev)
    ws_a = torch.empty(lc.accumulate_workspace_size(L, nb, d, act), dtype=torch.uint8, device=dev)
    ws_g = torch.empty(lc.gram_cross_workspace_size(), dtype=torch.uint8, device=dev)
    ws_s = torch.empty(lc.ridge_solve_workspace_size(L, d, k), dtype=torch.uint8, device=dev)
    names = ["error", "targets", "statistics", "step", "ridge_solve"]

    def step(ev=None):
        t = {n: 0.0 for n in names}
        marks = []

        def mark(n):
            if ev is not None:
                e = torch.cuda.Event(enable_timing=True)
                e.record(stream)
                marks.append((n, e))

        mark("start")
        lc.loca_error(z, cols, y, E, ce=ce, stream=stream)
        mark("error")
        if mb == 1:
            lc.loca_targets(E, P, Q, T, tsq=tsq, workspace=ws_t, stream=stream)
            mark("targets")
            lc.loca_gram_cross(X, T, ones, gram, cross, zero_first=True, workspace=ws_g, stream=stream)
            mark("statistics")
            lc.loca_step_from_gram(gram, tsq, w.eta, xsq, alpha, stream=stream)
            mark("step")
            lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, cross_scale=alpha,
                                workspace=ws_s, stream=stream)
        else:
            for m in range(mb):
                lc.loca_targets(E[m * nb:(m + 1) * nb], P, Q, T, tsq=tsq, workspace=ws_t, stream=stream)
                mark("targets")
                lc.loca_accumulate(X[m], T, tsq, w.eta, gram, cross, xsq, zero_first=(m == 0), workspace=ws_a,
                                   stream=stream)
                mark("statistics")
            mark("step")
            lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, workspace=ws_s, stream=stream)
        mark("ridge_solve")
        if ev is not None:
            ev.append((marks, t))

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    evs = []
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(steps):
        step(evs)
    b.record(stream)
    torch.cuda.synchronize()
    if lc.loca_device_status() != 0 or int(info.abs().sum().item()) != 0:
        raise SystemExit(f"{name}: a device error or a non-PD system")
    ms = a.elapsed_time(b) / steps
    stages = {n: 0.0 for n in names}
    for marks, _ in evs:
        for (_, e0), (n1, e1) in zip(marks, marks[1:]):
            stages[n1] += e0.elapsed_time(e1) / steps
    out = {"L": L, "d": d, "N": N, "C": C, "V": w.V, "r": r, "k": k, "micro_batches": mb,
           "dtype": "bf16" if act == torch.bfloat16 else "f32",
           "value": N * L / (ms / 1e3), "unit": UNIT, "ms_per_step": ms, "stages_ms": stages,
           "solve_ms": stages["ridge_solve"], "steps": steps, "warmup": warmup}
    if act == torch.bfloat16:
        flops = L * (2.0 * N * d * d + N * d * (d + 1.0))
        ach = flops / (stages["statistics"] / 1e3) / 1e12
        out["gram_roofline"] = {"bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                                "frac": ach / peak, "kernel": "k_gram_cross_tc (+ k_gram_mirror)"
                                + (", k_sumsq / k_step per batch" if mb > 1 else ""),
                                "flops_per_step": flops}
    else:
        out["gram_path"] = "fp32 inputs: k_gram_cross_f32 (CUDA cores, fp64 accumulation)"
    zb = N * V_bytes(z)
    out["error_roofline"] = hbm_object(zb + N * C * 4, stages["error"], "k_head_error", hbm)
    out["error_roofline"]["graded"] = w.V > 64 * w.C  # launch-bound when the row holds only the labels
    out["targets_roofline"] = hbm_object(L * N * d * T.element_size(), stages["targets"], "k_targets_tc", hbm,
                                         wpeak)
    out["ridge_solve_roofline"] = hbm_object(2 * L * d * d * 4, stages["ridge_solve"],
                                             "k_project_tc + k_chol_gram, k_chol_factor, k_chol_rows (reads of Gram and cross)", hbm)
    del inp, X, z, T, gram, cross, E, ce, B
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return out


def V_bytes(z):
    return z.shape[1] * z.element_size()


# ----------------------------------------------------------------------------- GPU arm

def run_ridge_only(args, w, lc, dev):
    """loca_ridge_solve alone at the workload's shape: seeded statistics (a Gram stand-in with a
    dominant diagonal, a dense cross product), W untimed and K timed calls on one stream; one JSON
    line.  The ridge solve's kernels run exactly as inside the step."""
    import torch

    L, d, k = w.L, w.d, w.k
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    gram = torch.randn((L, d, d), generator=g, device=dev)
    gram += float(d) * torch.eye(d, device=dev)
    cross = torch.randn((L, d, d), generator=g, device=dev)
    A = torch.randn((L, d, k), generator=g, device=dev) / float(d) ** 0.5
    nl = len(w.lambda_rel)
    B = torch.empty((nl, L, d, k), device=dev)
    info = torch.empty((nl, L), dtype=torch.int32, device=dev)
    xs = torch.full((L,), float(d) * d, dtype=torch.float64, device=dev)
    ws = torch.empty(lc.ridge_solve_workspace_size(L, d, k), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xs, workspace=ws, stream=stream)
    torch.cuda.synchronize()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(args.steps):
        lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xs, workspace=ws, stream=stream)
    b.record(stream)
    torch.cuda.synchronize()
    ms = a.elapsed_time(b) / args.steps
    byts = 2.0 * L * d * d * 4
    print(json.dumps({"ridge_only": w.name, "L": L, "d": d, "k": k, "nl": nl, "ms": ms,
                      "gbs_of_statistics": byts / (ms / 1e3) / 1e9, "status": lc.loca_device_status()}))


def main():
    args = parse()
    from synth import inputs as S

    w = S.WORKLOADS[args.workload]
    if args.L is not None or args.N is not None:
        w = S.scaled(w, L=args.L or w.L, N=args.N or w.N)
    if args.impl == "reference":
        rank = int(os.environ.get("RANK", "0"))
        if rank == 0:
            run_reference(args, w)
        return

    world0 = int(os.environ.get("WORLD_SIZE", "1"))
    rank0 = int(os.environ.get("RANK", "0"))
    host_info, tiny_times = None, None
    if rank0 == 0 and world0 == 1 and not args.no_cpu_baseline:
        # host-side only, before this process touches the GPU
        host_info = host_cpu()
        tiny_times = tiny_oracle_times()

    import numpy as np
    import torch

    world, rank, local = dist_setup(args)
    import __graft_entry__

    __graft_entry__.build()
    from paper_2608_03020_gb300 import loca as lc

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if args.ridge_only:
        run_ridge_only(args, w, lc, dev)
        return
    inp = S.device_inputs(w, seed=rank, device=dev)
    X, z, y, cols, P, Q, A = (inp[k] for k in ("X", "z", "y", "label_cols", "P", "Q", "A"))
    L, N, d, C, r, k = w.L, w.N, w.d, w.C, w.r, w.k
    nl = len(w.lambda_rel)
    act = X.dtype
    f32 = dict(dtype=torch.float32, device=dev)
    E = torch.empty((N, C), **f32)
    ce = torch.empty((N,), **f32)
    T = torch.empty((L, N, d), dtype=act, device=dev)
    tsq = torch.empty((L,), dtype=torch.float64, device=dev)
    xsq = torch.empty((L,), dtype=torch.float64, device=dev)
    alpha = torch.empty((L,), **f32)
    gram = torch.empty((L, d, d), **f32)
    cross = torch.empty((L, d, d), **f32)
    B = torch.empty((nl, L, d, k), **f32)
    info = torch.empty((nl, L), dtype=torch.int32, device=dev)
    ws_t = torch.empty(lc.targets_workspace_size(N, L, d), dtype=torch.uint8, device=dev)
    ones = torch.ones((L,), **f32)
    ws_g = torch.empty(lc.gram_cross_workspace_size(), dtype=torch.uint8, device=dev)
    ws_s = torch.empty(lc.ridge_solve_workspace_size(L, d, k), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    # k_head_error; k_targets_tc + k_reduce_partials; k_gram_cross_tc + k_gram_mirror; k_step_from_gram;
    # k_project_prep + k_project_tc + k_chol_gram + k_chol_factor + k_chol_rows
    launches_per_step = 1 + 2 + 2 + 1 + 5

    def step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        lc.loca_error(z, cols, y, E, ce=ce, stream=stream)
        if ev is not None:
            ev[1].record(stream)
        lc.loca_targets(E, P, Q, T, tsq=tsq, workspace=ws_t, stream=stream)
        if ev is not None:
            ev[2].record(stream)
        # one mini-batch: the cross product at alpha = 1, the step from the Gram trace, alpha
        # applied to the cross product in the solve (X is read by the Gram kernel only)
        lc.loca_gram_cross(X, T, ones, gram, cross, zero_first=True, workspace=ws_g, stream=stream)
        if ev is not None:
            ev[3].record(stream)
        lc.loca_step_from_gram(gram, tsq, w.eta, xsq, alpha, stream=stream)
        if ev is not None:
            ev[4].record(stream)
        lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, cross_scale=alpha,
                            workspace=ws_s, stream=stream)
        if ev is not None:
            ev[5].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    status = lc.loca_device_status()
    if status != 0:
        raise SystemExit(f"device status {status} after warm-up")
    # this GPU's write-only HBM rate in this run (a fill of T's 26 GB), the ceiling of the targets
    # kernel, whose traffic is the write of T
    wpeak = write_peak(T, stream)

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(args.steps)]
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        uuid = None
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clk:
        t_start = torch.cuda.Event(enable_timing=True)
        t_end = torch.cuda.Event(enable_timing=True)
        t_start.record(stream)
        for i in range(args.steps):
            step(evs[i])
        t_end.record(stream)
        torch.cuda.synchronize()
    barrier(world)
    ms_total = t_start.elapsed_time(t_end)
    ms_total = max_over_ranks(world, ms_total)
    ms_step = ms_total / args.steps
    stage_names = ["error", "targets", "gram_cross", "step", "ridge_solve"]
    stages = {n: statistics.mean(e[i].elapsed_time(e[i + 1]) for e in evs) for i, n in enumerate(stage_names)}
    status = lc.loca_device_status()
    if status != 0:
        raise SystemExit(f"device status {status} after the timed steps")
    if int(info.abs().sum().item()) != 0:
        raise SystemExit("a ridge system was not positive definite")
    value = world * N * L / (ms_step / 1e3)

    # roofline of the Gram / cross kernel
    peak, peak_kind = peaks()
    flops = L * (2.0 * N * d * d + N * d * (d + 1.0))
    achieved = flops / (stages["gram_cross"] / 1e3) / 1e12
    traffic = recorded_traffic(GRAM_TC_TRAFFIC, "gram_tc.cu", L, N=N, d=d)
    roofline = {"bound": "tensor", "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                "frac": achieved / peak, "traffic": traffic, "kernel": "k_gram_cross_tc",
                "peak_kind": f"bf16 dense sustained, {peak_kind}", "flops_per_launch": flops}
    hbm = hbm_peak()
    targets_roofline = hbm_object(L * N * d * T.element_size(), stages["targets"], "k_targets_tc", hbm, wpeak)
    targets_roofline["traffic"] = recorded_traffic(TARGETS_TRAFFIC, "targets.cu", L, N=N, d=d, r=r)
    solve_roofline = hbm_object(2 * L * d * d * 4, stages["ridge_solve"],
                                "k_project_tc + k_chol_gram, k_chol_factor, k_chol_rows (reads of Gram and cross)", hbm)
    solve_roofline["traffic"] = recorded_traffic(PROJECT_TRAFFIC, "project_tc.cu", L, d=d, k=k)
    solve_roofline["traffic_kernel"] = "k_project_tc"

    # the paper's own k-space statistics on the same inputs (no T, no d x d statistics):
    # error -> k-space accumulate (X A_l on the tensor cores, one HBM read of X) -> k-space solve
    kspace = None
    if not args.no_kspace:
        G_k = torch.empty((L, k, k), **f32)
        SC_k = torch.empty((L, C, k), **f32)
        xsq_k = torch.empty((L,), dtype=torch.float64, device=dev)
        B_k = torch.empty((nl, L, d, k), **f32)
        info_k = torch.empty((nl, L), dtype=torch.int32, device=dev)
        ws_k = torch.empty(lc.kspace_workspace_size(L, N, d, k, C, r), dtype=torch.uint8, device=dev)

        def kstep(ev=None):
            if ev is not None:
                ev[0].record(stream)
            lc.loca_error(z, cols, y, E, ce=ce, stream=stream)
            if ev is not None:
                ev[1].record(stream)
            lc.loca_kspace_accumulate(X, A, E, P, Q, w.eta, G_k, SC_k, xsq_k, zero_first=True, workspace=ws_k,
                                      stream=stream)
            if ev is not None:
                ev[2].record(stream)
            lc.loca_kspace_solve(G_k, SC_k, P, Q, w.lambda_rel, B_k, info_k, xsq_total=xsq_k, stream=stream)
            if ev is not None:
                ev[3].record(stream)

        for _ in range(args.warmup):
            kstep()
        torch.cuda.synchronize()
        kev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
        barrier(world)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(args.steps):
            kstep(kev[i])
        b.record(stream)
        torch.cuda.synchronize()
        ms_k = max_over_ranks(world, a.elapsed_time(b)) / args.steps
        if lc.loca_device_status() != 0 or int(info_k.abs().sum().item()) != 0:
            raise SystemExit("the k-space steps reported a device error or a non-PD system")
        kst = {n: statistics.mean(e[i].elapsed_time(e[i + 1]) for e in kev)
               for i, n in enumerate(["error", "accumulate", "solve"])}
        xbytes = float(X.numel() * X.element_size())
        kspace = {"value": world * N * L / (ms_k / 1e3), "unit": UNIT, "ms_per_step": ms_k, "stages_ms": kst,
                  "launches_per_step": 1 + 4 + 1,
                  "roofline": {"bound": "hbm", "achieved": xbytes / (kst["accumulate"] / 1e3) / 1e9,
                               "peak": hbm_peak(), "unit": "GB/s",
                               "frac": xbytes / (kst["accumulate"] / 1e3) / 1e9 / hbm_peak(),
                               "traffic": recorded_traffic(KSPACE_TRAFFIC, "kspace.cu", L, N=N, d=d, k=k),
                               "traffic_kernel": "k_kspace_xa",
                               "kernel": "loca_kspace_accumulate (prep, X A on tcgen05, stats, final)",
                               "bytes_per_launch": xbytes}}

    # the same pass with the targets generated inside the statistics kernel (T never written):
    # error -> ||T||^2 in closed form -> fused Gram / cross at alpha = 1 -> step -> solve
    fused = None
    if not args.no_fused and X.dtype == torch.bfloat16:
        tsq_f = torch.empty((L,), dtype=torch.float64, device=dev)
        ws_q = torch.empty(lc.targets_sq_workspace_size(N, C), dtype=torch.uint8, device=dev)
        ws_f = torch.empty(lc.gram_cross_fused_workspace_size(L, N, r), dtype=torch.uint8, device=dev)

        def fstep(ev=None):
            if ev is not None:
                ev[0].record(stream)
            lc.loca_error(z, cols, y, E, ce=ce, stream=stream)
            if ev is not None:
                ev[1].record(stream)
            lc.loca_targets_sq(E, P, Q, tsq_f, workspace=ws_q, stream=stream)
            if ev is not None:
                ev[2].record(stream)
            lc.loca_gram_cross_fused(X, E, P, Q, ones, gram, cross, zero_first=True, workspace=ws_f, stream=stream)
            if ev is not None:
                ev[3].record(stream)
            lc.loca_step_from_gram(gram, tsq_f, w.eta, xsq, alpha, stream=stream)
            if ev is not None:
                ev[4].record(stream)
            lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, cross_scale=alpha,
                                workspace=ws_s, stream=stream)
            if ev is not None:
                ev[5].record(stream)

        for _ in range(args.warmup):
            fstep()
        torch.cuda.synchronize()
        fev = [[torch.cuda.Event(enable_timing=True) for _ in range(6)] for _ in range(args.steps)]
        barrier(world)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for i in range(args.steps):
            fstep(fev[i])
        b.record(stream)
        torch.cuda.synchronize()
        ms_f = max_over_ranks(world, a.elapsed_time(b)) / args.steps
        if lc.loca_device_status() != 0 or int(info.abs().sum().item()) != 0:
            raise SystemExit("the fused-targets steps reported a device error or a non-PD system")
        fst = {n: statistics.mean(e[i].elapsed_time(e[i + 1]) for e in fev)
               for i, n in enumerate(["error", "targets_sq", "gram_cross_fused", "step", "ridge_solve"])}
        ach_f = flops / (fst["gram_cross_fused"] / 1e3) / 1e12
        fused = {"value": world * N * L / (ms_f / 1e3), "unit": UNIT, "ms_per_step": ms_f, "stages_ms": fst,
                 "vs_split": {"targets_plus_gram_ms": stages["targets"] + stages["gram_cross"],
                              "targets_sq_plus_fused_ms": fst["targets_sq"] + fst["gram_cross_fused"]},
                 "roofline": {"bound": "tensor", "achieved": ach_f, "peak": peak, "unit": "TFLOP/s",
                              "frac": ach_f / peak, "kernel": "k_gram_cross_tc<fused> (+ k_gram_mirror)",
                              "flops_per_launch": flops, "note": "useful flops of the statistics only; the "
                              "generation of T adds 6 N d r flops per block on the tensor cores"}}
        del ws_q, ws_f

    # the head error where it is HBM-bound: the Qwen2.5-14B row of the workloads (N = 131072 tokens,
    # V = 151936 bf16 logits, C = 4 label columns; 39.8 GB of logits, drawn as in synth)
    vocab = None
    if not args.no_vocab and world == 1:
        wv = S.WORKLOADS["qwen2.5-14b"]
        if args.vocab_N is not None:
            wv = S.scaled(wv, L=wv.L, N=args.vocab_N)
        gen = torch.Generator(device=dev)
        gen.manual_seed(1234)
        zv = torch.empty((wv.N, wv.V), dtype=torch.bfloat16, device=dev)
        rng = np.random.default_rng(1234)
        cols_v = torch.from_numpy(np.sort(rng.choice(wv.V, size=wv.C, replace=False)).astype(np.int32)).to(dev)
        y_v = torch.from_numpy(rng.integers(0, wv.C, wv.N).astype(np.int32)).to(dev)
        off = float(np.log(wv.V / wv.C))
        for n0 in range(0, wv.N, 8192):
            g = torch.randn((min(8192, wv.N - n0), wv.V), generator=gen, device=dev)
            g[:, cols_v.long()] += off
            zv[n0:n0 + g.shape[0]] = g.to(torch.bfloat16)
            del g
        Ev = torch.empty((wv.N, wv.C), **f32)
        cev = torch.empty((wv.N,), **f32)
        for _ in range(args.warmup):
            lc.loca_error(zv, cols_v, y_v, Ev, ce=cev, stream=stream)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.steps):
            lc.loca_error(zv, cols_v, y_v, Ev, ce=cev, stream=stream)
        b.record(stream)
        torch.cuda.synchronize()
        ms_v = a.elapsed_time(b) / args.steps
        zb = float(zv.numel() * zv.element_size())
        vocab = {"workload": "qwen2.5-14b head error", "N": wv.N, "V": wv.V, "C": wv.C, "ms": ms_v,
                 "roofline": {"bound": "hbm", "achieved": zb / (ms_v / 1e3) / 1e9, "peak": hbm_peak(), "unit": "GB/s",
                              "frac": zb / (ms_v / 1e3) / 1e9 / hbm_peak(), "kernel": "k_head_error<bf16>",
                              "bytes_per_launch": zb}}
        del zv, Ev, cev
        torch.cuda.empty_cache()

    # the one-shot feedback fit in the paper's d-wide error space (m = d) at the 7B width: every
    # block's rank-16 map from Np = 8192 probe pairs, randomized subspace iteration with a sketch
    # of 32 and two power iterations (untimed in the step; reported on its own)
    calib = None
    if not args.no_calib and world == 1:
        Np_c, m_c, r_c, ell_c, q_c = 8192, d, 16, 32, 2
        pc = S.device_probe_pairs(Np_c, m_c, d, L, rank=8, seed=1, device=dev)
        Ec, Gc = pc["E_probe"], pc["G_probe"]
        Om = torch.from_numpy(S.omega_matrix(d, ell_c, seed=1)).to(dev)
        beta_c = 1e-3 * float(torch.sum(Ec.double() ** 2).item()) / m_c
        Pc = torch.empty((L, m_c, r_c), **f32)
        Qc = torch.empty((L, r_c, d), **f32)
        wsc = torch.empty(lc.calib_fit_rsvd_workspace_size(Np_c, m_c, d, L, r_c, ell_c), dtype=torch.uint8,
                          device=dev)
        lc.loca_calib_fit_rsvd(Ec, Gc, beta_c, r_c, Om, q_c, Pc, Qc, workspace=wsc, stream=stream)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(3):
            lc.loca_calib_fit_rsvd(Ec, Gc, beta_c, r_c, Om, q_c, Pc, Qc, workspace=wsc, stream=stream)
        b.record(stream)
        torch.cuda.synchronize()
        if lc.loca_device_status() != 0:
            raise SystemExit("the feedback fit reported a device error")
        calib = {"workload": "qwen2.5-7b feedback fit, d-wide error space", "Np": Np_c, "m": m_c, "d": d, "L": L,
                 "r": r_c, "ell": ell_c, "q": q_c, "ms": a.elapsed_time(b) / 3,
                 "method": "randomized subspace iteration + Rayleigh-Ritz (loca_calib_fit_rsvd)"}
        del Ec, Gc, pc, wsc, Pc, Qc
        torch.cuda.empty_cache()

    # end to end through the public API: host inputs copied in, adapters copied out, per step
    e2e = None
    if not args.no_e2e:
        pin = dict(pin_memory=True)
        # X in loca_host_alloc memory (page-locked, 2 MiB pages): copies run at the link rate
        hX = lc.host_empty(X.shape, X.dtype)
        hX.copy_(X)
        hz = torch.empty(z.shape, dtype=z.dtype, **pin)
        hz.copy_(z)
        small = {kk: torch.empty(v.shape, dtype=v.dtype, **pin).copy_(v) for kk, v in
                 (("y", y), ("cols", cols), ("P", P), ("Q", Q), ("A", A))}
        hB = torch.empty(B.shape, dtype=B.dtype, **pin)
        hinfo = torch.empty(info.shape, dtype=info.dtype, **pin)
        h2d = sum(t.numel() * t.element_size() for t in [hX, hz, *small.values()])
        d2h = hB.numel() * hB.element_size() + hinfo.numel() * hinfo.element_size()

        # X streams from host memory through loca_accumulate_streamed: groups of `group` blocks
        # are copied into a two-slot device staging ring while the previous group's statistics run
        group = max(1, min(args.e2e_group, L))
        staging = torch.empty((2 * group, N, d), dtype=act, device=dev)
        ws_a = torch.empty(lc.accumulate_workspace_size(L, N, d, act), dtype=torch.uint8, device=dev)

        def e2e_step():
            z.copy_(hz, non_blocking=True)
            y.copy_(small["y"], non_blocking=True)
            cols.copy_(small["cols"], non_blocking=True)
            P.copy_(small["P"], non_blocking=True)
            Q.copy_(small["Q"], non_blocking=True)
            A.copy_(small["A"], non_blocking=True)
            lc.loca_error(z, cols, y, E, ce=ce, stream=stream)
            lc.loca_targets(E, P, Q, T, tsq=tsq, workspace=ws_t, stream=stream)
            lc.loca_accumulate_streamed(hX, staging, T, tsq, w.eta, gram, cross, xsq, zero_first=True,
                                        group=group, workspace=ws_a, stream=stream)
            lc.loca_ridge_solve(gram, cross, A, w.lambda_rel, B, info, xsq_total=xsq, workspace=ws_s,
                                stream=stream)
            hB.copy_(B, non_blocking=True)
            hinfo.copy_(info, non_blocking=True)

        e2e_steps = max(1, min(args.steps, 5))
        e2e_step()
        torch.cuda.synchronize()

        # the link's host-to-device rate right before the timed steps: the host memory and its
        # bandwidth are shared with whatever else runs on the machine
        def link_gbs():
            nb = min(group, L) * N * d
            a_, b_ = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a_.record(stream)
            staging.view(-1)[:nb].copy_(hX.view(-1)[:nb], non_blocking=True)
            b_.record(stream)
            torch.cuda.synchronize()
            return nb * staging.element_size() / (a_.elapsed_time(b_) / 1e3) / 1e9

        link_before = link_gbs()
        barrier(world)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(e2e_steps):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        ms_e2e = max_over_ranks(world, a.elapsed_time(b)) / e2e_steps
        link_after = link_gbs()
        e2e = {"value": world * N * L / (ms_e2e / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e, "steps": e2e_steps,
               "x_from_host": f"loca_accumulate_streamed, {group} blocks per copy",
               "h2d_link_gbs_before_after": [round(link_before, 1), round(link_after, 1)]}
        if int(info.abs().sum().item()) != 0 or lc.loca_device_status() != 0:
            raise SystemExit("the end-to-end steps reported a device error or a non-PD system")
        del hX, hz, staging

    x_gb = X.numel() * X.element_size() / 1e9
    # every other workload at its own shape (the headline's buffers released first)
    configs = None
    if not args.no_configs and world == 1:
        del X, z, T, gram, cross, inp, ws_t, ws_g, ws_s, B, E, ce
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        configs = {}
        for name in ("tiny", "qwen2.5-0.5b", "qwen2.5-1.5b", "smollm2-1.7b", "qwen2.5-14b"):
            if name == w.name:
                continue
            configs[name] = measure_workload(lc, name, dev, stream, max(1, min(args.steps, 5)), args.warmup, peak,
                                             hbm, wpeak)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # bounded sample: one block, a token prefix sized from a 2048-token pilot run to take about
        # 15 s of CPU time (capped at the full N)
        pilot = min(2048, N)
        host = host_sample(w, tokens=pilot)
        oracle_sample(w, min(512, pilot), host)
        per_token = oracle_sample(w, pilot, host) / pilot
        tokens = int(min(N, max(pilot, (15.0 / max(per_token, 1e-9)) // 1024 * 1024)))
        host = host_sample(w, tokens=tokens)
        sec = oracle_sample(w, tokens, host)
        cpu = {"value": tokens / sec, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle",
               "sample": f"one block (of {L}), first {tokens} of {N} tokens, full d={d}, C={C}, r={r}, k={k}; "
                         f"numpy fp64, {sec:.1f} s",
               "host": host_info, "tiny_workload_full_pass": tiny_times}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "L": L, "d": d, "N": N, "C": C, "r": r, "k": k,
                       "lambda_rel": list(w.lambda_rel), "eta": w.eta, "parallelism": f"replicas{world}",
                       "l2": "inputs larger than L2 (X is %.1f GB)" % x_gb},
            "stages_ms": stages,
            "solve_ms": stages["ridge_solve"],
            "roofline": roofline,
            "targets_roofline": targets_roofline,
            "ridge_solve_roofline": solve_roofline,
            "write_peak_gbs": wpeak,
            "configs": configs,
            "gpu_launches": launches_per_step * args.steps,
            "e2e": e2e,
            "kspace": kspace,
            "fused_targets": fused,
            "head_error_vocab": vocab,
            "calibration": calib,
            "cpu_baseline": cpu,
            "clocks": clk.summary(),
        }
        print(json.dumps(line))
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


if __name__ == "__main__":
    main()
