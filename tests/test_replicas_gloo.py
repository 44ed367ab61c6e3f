"""The multi-GPU path is replicas only (one independent denoise per rank, no data-path
collective). Its host logic runs here as world-size-2 gloo ranks on the CPU: max-over-ranks
timing, the whole-job rate, independent per-rank requests, and the reference arm printing one
line from rank 0 under torchrun."""

import hashlib
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


def _rank(rank, world, port, q):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    from synth import TINY, make_requests
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    slowest = bench.max_over_ranks(10.0 + 5.0 * rank, world, "cpu")
    r = make_requests(TINY, bench.request_seed(rank), 1, 8, 4)
    digest = hashlib.sha256(r["noise"].tobytes() + r["prefix_k"].tobytes()).hexdigest()
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, slowest, digest))


def test_two_gloo_ranks_take_the_slowest_time_and_own_requests():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [x[1] for x in res] == [15.0, 15.0]          # both ranks see the slowest rank's time
    assert res[0][2] != res[1][2]                        # each rank denoises its own requests


def test_whole_job_rate_counts_every_replica():
    sys.path.insert(0, ROOT)
    import bench
    one = bench.whole_job_rate(1, 4, 10, 50.0)
    assert one == pytest.approx(4 * 10 / 0.05)
    assert bench.whole_job_rate(2, 4, 10, 50.0) == pytest.approx(2 * one)
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5


def test_reference_arm_under_torchrun_prints_once():
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "1",
           "--warmup", "3"]
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["value"] > 0
