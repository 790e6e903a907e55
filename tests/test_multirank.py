"""The benchmark's multi-GPU path on CPU: two gloo ranks (one process each,
as torchrun launches them) agree on the slowest rank's timed region, and the
whole-job rate counts every rank's pack (weak scaling: members are
independent, each rank trains its own pack and no collective touches the
data path).  The reference arm under torchrun prints from rank 0 only."""
import os
import socket
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ms = bench.max_over_ranks(100.0 + 7.5 * rank, dist, "cpu")
    out[rank] = (ms, bench.job_rate(world, 32, 512, 10, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_share_the_slowest_time():
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(2, port, out), nprocs=2, join=True)
        res = dict(out)
    assert res[0] == res[1]
    ms, rate = res[0]
    assert ms == 107.5
    assert rate == pytest.approx(2 * 32 * 512 * 10 / 0.1075)


def test_reference_arm_prints_from_rank_zero_only():
    """`bench.py --impl reference` under torchrun: rank 1 exits without
    output, rank 0 prints one JSON line (a tiny sample of the CPU oracle)."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={port}", os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3", "--workload", "tiny"]
    env = dict(os.environ, OMP_NUM_THREADS="2")
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    import json
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0


def test_reference_arm_fits_its_time_budget():
    """`bench.py --impl reference` times exactly K oracle steps and sizes
    each step's rows so that W + K steps fit the budget: with K = 400 and a
    4 s budget on the tiny workload the rows are cut below the batch (on a
    host fast enough for 400 full steps in 4 s they are not) and the run ends
    in seconds."""
    import json
    import time
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "400", "--warmup", "3",
           "--workload", "tiny", "--reference-seconds", "4"]
    t0 = time.perf_counter()
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=ROOT)
    wall = time.perf_counter() - t0
    assert r.returncode == 0, r.stderr[-2000:]
    d = json.loads(r.stdout.strip().splitlines()[-1])
    assert d["impl"] == "reference" and d["steps"] == 400 and d["value"] > 0
    sample = d["cpu_baseline"]["sample"]
    assert "400 timed steps of" in sample and ("to fit the time budget" in sample or "the full batch" in sample)
    # the same config keys as the GPU arm's line
    assert set(d["config"]) == {"workload", "params", "gemm_flop_per_step", "l2", "parallelism", "batches",
                                "optimizer", "embeddings"}
    assert d["e2e"]["h2d_bytes_per_step"] == 0
    assert wall < 120, wall
