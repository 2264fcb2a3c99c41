"""The multi-rank path of the benchmark on CPU (gloo, world size 2): the job's
time is its slowest rank's, its throughput counts every rank's tape, and
the reference arm runs on rank 0 alone (a non-zero rank exits cleanly without
work).  No GPU is involved."""
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


def _worker(rank, ws, port, times, out):
    import torch.distributed as dist

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    sys.path.insert(0, ROOT)
    dist.init_process_group("gloo", rank=rank, world_size=ws)
    import bench

    out.put((rank, bench.max_over_ranks(times[rank], ws, "cpu")))
    dist.barrier()
    dist.destroy_process_group()


def test_slowest_rank_sets_the_time_gloo():
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    q = mp.Queue()
    times = [3.25, 5.5]
    port = _free_port()
    procs = [mp.Process(target=_worker, args=(r, 2, port, times, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    assert got == {0: 5.5, 1: 5.5}


def test_job_throughput_counts_every_rank():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(2.5, 1, "cpu") == 2.5
    assert bench.job_throughput(1, 1 << 20, 2.0) == pytest.approx((1 << 20) / 2e-3)
    assert bench.job_throughput(4, 1 << 20, 2.0) == pytest.approx(4 * (1 << 20) / 2e-3)


def test_reference_arm_runs_on_rank_zero_only():
    # a non-zero rank of a torchrun job (RANK / WORLD_SIZE as torchrun sets them) exits 0
    # at once and prints nothing; rank 0 alone times the oracle and prints the line
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2", MASTER_ADDR="127.0.0.1",
               MASTER_PORT=str(_free_port()))
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "1",
           "--warmup", "3"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=ROOT, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    assert not [l for l in r.stdout.splitlines() if l.startswith("{")]
