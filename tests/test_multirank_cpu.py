"""The multi-rank plumbing of bench.py on CPU (world size 2, gloo, 127.0.0.1; no GPU needed).

The method needs one GPU and no collective; ``bench.py --gpus N`` runs N independent replicas
whose only exchange is the timing reduction (max over ranks) and barriers.  Checked here:
rank set-up from the torchrun environment, the barrier, the max-over-ranks reduction, and
that under torchrun the reference arm prints exactly one JSON line (rank 0) while every rank
exits 0.
"""

import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _cpu_env(port):
    env = dict(os.environ)
    env.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), CUDA_VISIBLE_DEVICES="")
    env["PYTHONPATH"] = ROOT + os.pathsep + env.get("PYTHONPATH", "")
    return env


RANK_SCRIPT = r"""
import json, os, sys
sys.path.insert(0, os.environ["ROOT"])
import bench
class A: pass
world, rank, local = bench.dist_setup(A())
bench.barrier(world)
m = bench.max_over_ranks(world, 1.5 + rank)
bench.barrier(world)
print(json.dumps({"rank": rank, "world": world, "max": m}))
import torch.distributed as dist
dist.destroy_process_group()
"""


def test_rank_setup_barrier_and_max_over_ranks():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = _cpu_env(port)
        env.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2", ROOT=ROOT)
        procs.append(subprocess.Popen([sys.executable, "-c", RANK_SCRIPT], env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=120)
        assert p.returncode == 0, err[-2000:]
        outs.append(json.loads(out.strip().splitlines()[-1]))
    assert sorted(o["rank"] for o in outs) == [0, 1]
    assert all(o["world"] == 2 and o["max"] == 2.5 for o in outs)


def test_reference_arm_under_torchrun_prints_one_line():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"), "--impl", "reference",
           "--workload", "tiny", "--gpus", "2", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, env=_cpu_env(port), capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["value"] > 0 and line["n_gpus"] == 2
