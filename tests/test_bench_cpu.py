"""The benchmark's CPU legs (the cpu_baseline and the --impl reference arm
run the oracle on the host): every workload defines the methods the bench
calls, and small instances of the replay workloads run their oracle rounds,
so a broken CPU leg shows up here rather than on the GPU machine."""
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

METHODS = ["config", "setup", "schedules", "deliver_once", "latency_step",
           "e2e_setup", "e2e_round", "cpu_setup", "cpu_round"]


@pytest.mark.parametrize("name", sorted(bench.WORKLOADS) + ["sharded-" + n for n in
                                                            sorted(bench.SHARDED)])
def test_workload_has_every_leg(name):
    if name.startswith("sharded-"):
        wl = bench.SHARDED[name[len("sharded-"):]](rank=1)
    else:
        wl = bench.WORKLOADS[name]()
    for m in METHODS:
        assert callable(getattr(wl, m, None)), (name, m)
    for attr in ("kernel", "dtype", "deliver_bytes", "round_bytes", "launches_per_round"):
        assert hasattr(wl, attr), (name, attr)


class _SmallGrpo(bench.LlmBatch):
    P, G = 8, 4


@pytest.mark.parametrize("make,kw", [
    (lambda: bench.PerReplay(capacity=4096, batch=16), {"host_frames": 512}),
    (lambda: bench.MmReplay(capacity=64, batch=8), {"host_rows": 16}),
    (lambda: bench.MmReplay(capacity=64, batch=8, hbm_frac=0.5, ingest=4), {"host_rows": 16}),
    (lambda: bench.DqnTiny(capacity=256, batch=8), {}),
    (lambda: bench.PpoIteration(), {}),
    (lambda: _SmallGrpo(), {}),
])
def test_cpu_rounds_run(make, kw):
    wl = make()
    wl.cpu_setup(**kw)
    assert isinstance(wl.cpu_sample, str) and wl.cpu_sample
    for r in range(3):
        wl.cpu_round(r)
