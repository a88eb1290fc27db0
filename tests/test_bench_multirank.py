"""The N > 1 path of bench.py on the host: world-size-2 gloo process groups on CPU.

Each rank runs its own replica (sessions are independent, no collective on the data
path); the only cross-rank steps are the timing barrier and the reductions of the
whole-job throughput, and, for the reference arm, that rank 0 alone works and prints."""
import json
import os
import socket
import subprocess
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # Rank r processed 10 (r + 1) units in 100 (r + 1) ms.
        v, ms = bench.job_throughput(10.0 * (rank + 1), 100.0 * (rank + 1), world)
        dist.barrier()
        results[rank] = (v, ms)
    finally:
        dist.destroy_process_group()


def test_job_throughput_sums_units_over_the_slowest_rank():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        results = m.dict()
        mp.spawn(_rank_main, args=(world, port, results), nprocs=world, join=True)
        got = dict(results)
    # (10 + 20) units over the slowest rank's 200 ms, the same on every rank.
    for rank in range(world):
        v, ms = got[rank]
        assert ms == pytest.approx(200.0)
        assert v == pytest.approx(30.0 / 0.2)


def test_job_throughput_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_throughput(64.0, 50.0, 1) == (pytest.approx(1280.0), 50.0)


def test_reference_arm_under_torchrun_prints_once_from_rank_0():
    port = _free_port()
    r = subprocess.run(
        [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
         "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl",
         "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"],
        cwd=ROOT, capture_output=True, text=True, timeout=900,
        env=dict(os.environ, CUDA_VISIBLE_DEVICES="", OMP_NUM_THREADS="4"))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
