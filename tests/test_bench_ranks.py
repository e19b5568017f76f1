"""The multi-rank (N > 1) bench path, on CPU with gloo ranks.

With N GPUs the benchmark runs N independent replicas of the experience path
(nothing is exchanged on the data path), brackets the timed region with a
barrier, takes the maximum time over ranks and reports the whole-job
throughput of all replicas.  Here two gloo ranks on 127.0.0.1 run the same
reduction and throughput helpers that the bench uses with NCCL, and the
reference arm is checked to leave every rank but rank 0 without work.
"""
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


def _rank_main(rank, world, port, times, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        ms = bench.job_ms(times[rank], dist, torch.device("cpu"))
        gbs = bench.job_gbs(1e9, 10, world, ms)
        out.put((rank, ms, gbs))
        dist.barrier()
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_gloo_ranks_take_max_time_and_sum_work():
    world, times = 2, [12.5, 40.0]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, times, out))
             for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=100) for _ in range(world))
    for p in procs:
        p.join(timeout=30)
        assert p.exitcode == 0
    for rank, ms, gbs in res:
        assert ms == 40.0, rank  # the slowest replica bounds the job
        # 2 ranks x 10 steps x 1 GB in 40 ms
        assert gbs == pytest.approx(2 * 10 * 1.0 / 0.040)


def test_job_helpers_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_ms(7.0, None, None) == 7.0
    assert bench.job_gbs(2e9, 5, 1, 1000.0) == pytest.approx(10.0)


def test_reference_arm_non_zero_rank_does_no_work():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    p = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl",
                        "reference", "--gpus", "2", "--steps", "3", "--warmup", "3"],
                       env=env, capture_output=True, text=True, timeout=120)
    assert p.returncode == 0, p.stderr
    assert p.stdout.strip() == ""
