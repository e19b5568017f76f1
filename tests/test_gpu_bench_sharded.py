"""bench.py's N > 1 path for the sharded workloads, launched as the driver
launches it (torch.distributed.run, one process per rank), with two ranks
sharing the one GPU: the gloo backend stages every exchange through host
memory, so no kernel of one rank waits on another's.  Each run must print one
JSON line from rank 0 with the whole-job throughput of both ranks and the
sharded parallelism."""
import json
import os
import socket
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.timeout(600)
@pytest.mark.parametrize("workload,extra", [("per1m", ["--capacity", "20000"]),
                                            ("ppo", [])])
def test_bench_sharded_two_ranks_on_one_gpu(workload, extra):
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes", "1",
           "--nproc-per-node", "2", "--master-addr", "127.0.0.1", "--master-port",
           str(_free_port()), "bench.py", "--gpus", "2", "--workload", workload,
           "--dist-backend", "gloo", "--steps", "4", "--warmup", "3", "--no-cpu-baseline",
           "--no-extra", "--kernel-steps", "3", "--latency-steps", "3", "--e2e-steps", "3"
           ] + extra
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=540)
    assert p.returncode == 0, p.stderr[-3000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, p.stdout[-2000:]
    line = json.loads(lines[0])
    assert line["n_gpus"] == 2
    assert line["config"]["parallelism"] == "sharded2"
    assert line["config"]["workload"].endswith("-sharded")
    assert line["value"] > 0 and line["e2e"]["value"] > 0
    assert line["gpu_launches"] > 0
