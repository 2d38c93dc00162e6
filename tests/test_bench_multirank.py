"""The N > 1 path of bench.py on CPU with world-size-2 gloo ranks: every rank
draws its own batch, the step time is the slowest rank's, the whole-job
throughput counts the tokens of all ranks, and under torchrun the reference arm
runs on rank 0 alone and prints exactly one JSON line."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import torch.multiprocessing as mp

import bench
from paper_2609_26590_gb300 import workloads as wl

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    import torch.distributed as dist
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 1.0 + 2.5 * rank                 # rank 1 is the slow one
        dist.barrier()
        slowest = bench.max_over_ranks(local_ms, dist, "cpu")
        w = wl.WORKLOADS[0]
        inp = wl.workload_inputs(w, seed=bench.rank_seed(w, rank))
        with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
            json.dump({"slowest": slowest, "q0": float(inp["q"].reshape(-1)[0]),
                       "seed": bench.rank_seed(w, rank)}, f)
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_per_rank_batches_gloo(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn")
    r = [json.load(open(tmp_path / f"rank{i}.json")) for i in range(world)]
    assert r[0]["slowest"] == r[1]["slowest"] == 3.5      # both ranks see the max
    assert r[0]["seed"] != r[1]["seed"]                  # independent batches
    assert r[0]["q0"] != r[1]["q0"]
    # whole-job throughput: tokens of all ranks over the slowest rank's step time
    assert bench.job_tokens_per_s(1600, world, 2.0) == 2 * 1600 / 2.0e-3
    assert bench.max_over_ranks(1.25, None, "cpu") == 1.25


def test_reference_arm_under_torchrun_prints_once():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "1", "--workload", "0"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and np.isfinite(d["ms_per_step"])


def test_sswiglu_reference_arm_prints_one_line():
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--op", "sswiglu",
           "--sw-workload", "0", "--steps", "1", "--warmup", "1"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
    assert d["config"]["workload"] == "sswiglu_tiny_8x12" and d["e2e"]["h2d_bytes_per_step"] == 0
