"""The multi-replica path of bench.py on CPU: world_size-2 gloo process groups.

On N GPUs bench.py runs N independent replicas (the path has no data-path
collective); the ranks meet only at the timing barrier and the max-over-ranks
reduction, and the whole-job value is N x the per-rank work / the slowest
rank's time. Those host steps are checked here with the gloo backend."""
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # per-rank step and dominant-kernel times (ms): rank 1 is the slower one for the step,
        # rank 0 for the kernel
        got = bench.max_over_ranks([1.0 + rank, 0.5 - 0.25 * rank], world, "cpu")
        dist.barrier()
        q.put((rank, got, bench.dist_setup()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_rank_and_scale_the_job_value():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, setup in out:
        assert got == [2.0, 0.5]  # element-wise max over the ranks, on every rank
        assert setup == (world, rank, rank)
    import bench
    # whole-job value: both replicas' work over the slowest rank's time
    assert bench.job_tflops(2, 1e12, 2.0e-3) == pytest.approx(1000.0)
    assert bench.max_over_ranks([3.0], 1, "cpu") == [3.0]


def test_reference_arm_runs_on_rank_zero_only():
    # under torchrun the oracle arm runs on rank 0; another rank exits 0 without work or output
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], env=env, capture_output=True, text=True, timeout=120, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""
