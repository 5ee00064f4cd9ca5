"""The N > 1 host logic of bench.py on CPU ranks (gloo, world size 2): the
replicas share nothing but the timing reduction (max over ranks), the
whole-job value counts every rank's images, and the reference arm runs on
rank 0 only."""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r "took" 100 (r + 1) ms for 5 steps of 256 images
        total, value = bench.whole_job_rate(dist, 100.0 * (rank + 1), 256 * 5, world, device="cpu")
        q.put((rank, total, value))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_all_images():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = {}
    try:
        for _ in range(2):
            rank, total, value = q.get(timeout=120)
            out[rank] = (total, value)
    finally:
        for p in procs:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    assert all(p.exitcode == 0 for p in procs)
    for rank in (0, 1):
        total, value = out[rank]
        assert total == 200.0                       # the slower rank's timed region
        assert value == pytest.approx(2 * 256 * 5 / 0.2)  # both ranks' images / that time


def test_single_rank_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    total, value = bench.whole_job_rate(None, 50.0, 100, 1)
    assert (total, value) == (50.0, 2000.0)


def test_reference_arm_runs_on_rank_0_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                        "--warmup", "0"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""
