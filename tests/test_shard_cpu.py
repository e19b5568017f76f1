"""The host side of the sharded buffer, on the CPU.

1. ShardComm's collectives on two gloo ranks (127.0.0.1): all-gather in rank
   order, all-to-all with uneven splits of multi-dimensional rows (the
   learner's batch travels this way), in-place sum and minimum.
2. The reading the sharded path rests on: the stratified targets of one
   buffer whose leaves are the shards' leaves in shard-major order, routed
   to the shard whose prefix range holds them and found there by the shard's
   own inverse CDF, give the global inverse CDF's answer; the routed
   targets never decrease, so grouping them by owner keeps stratum order.
   Checked with the oracle's sampler, target rule and Philox on random
   shards, including empty shards and zero priorities.
3. A rank that leaves between rounds: the survivor's next exchange ends in
   an error within the process group's timeout, not in an endless wait.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _comm_rank(rank, world, port, out):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2609_24456_gb300.shard import ShardComm
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        c = ShardComm()
        res = {"rank": c.rank, "world": c.world, "host": c.host}
        res["gather"] = c.all_gather(torch.tensor([10 * rank, 10 * rank + 1])).tolist()
        # rank 0 sends 1 row to 0 and 2 to 1; rank 1 sends 3 rows to 0 and 0 to 1
        send = [[1, 2], [3, 0]][rank]
        recv = [send_r[rank] for send_r in ([1, 2], [3, 0])]
        rows = torch.arange(sum(send) * 6, dtype=torch.float32).reshape(-1, 2, 3) + 100 * rank
        res["a2a"] = c.all_to_all(rows, send, recv).tolist()
        buf = torch.full((5, 2, 3), -1.0)
        c.all_to_all(rows, send, recv, out=buf)
        res["a2a_out"] = buf.tolist()
        s = torch.tensor([0.5 + rank, 2.0], dtype=torch.float64)
        res["sum"] = c.all_reduce(s, "sum").tolist()
        m = torch.tensor([7 - rank], dtype=torch.int64)
        res["min"] = c.all_reduce(m, "min").tolist()
        out.put(res)
    finally:
        dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_shard_comm_on_two_gloo_ranks():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_comm_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=100) for _ in range(world)), key=lambda d: d["rank"])
    for p in procs:
        p.join(timeout=30)
        assert p.exitcode == 0
    rows = [np.arange(18, dtype=np.float32).reshape(-1, 2, 3),
            np.arange(18, dtype=np.float32).reshape(-1, 2, 3) + 100]
    # rank 0 gets row 0 of rank 0, then rows 0..2 of rank 1; rank 1 gets
    # rows 1..2 of rank 0
    want = [np.concatenate([rows[0][:1], rows[1][:3]]), rows[0][1:3]]
    for r, d in enumerate(res):
        assert d["world"] == 2 and d["host"]
        assert d["gather"] == [0, 1, 10, 11]
        assert np.array_equal(np.array(d["a2a"]), want[r])
        got = np.array(d["a2a_out"])
        assert np.array_equal(got[:len(want[r])], want[r])
        assert (got[len(want[r]):] == -1).all()
        assert d["sum"] == [2.0, 4.0]
        assert d["min"] == [6]


def _inverse_cdf(leaves, t):
    """The i with prefix(i) <= t < prefix(i) + q_i (brute force)."""
    acc = 0
    for i, q in enumerate(leaves):
        if acc <= t < acc + int(q):
            return i
        acc += int(q)
    raise AssertionError("target beyond the total")


@pytest.mark.parametrize("case", range(6))
def test_routing_by_shard_prefix_is_the_global_inverse_cdf(orc, case):
    rng = np.random.default_rng(100 + case)
    G = int(rng.integers(1, 6))
    shards = []
    for g in range(G):
        n = int(rng.integers(1, 40))
        q = rng.integers(0, 5000, size=n).astype(np.uint32)
        q[rng.random(n) < 0.3] = 0
        if rng.random() < 0.25:
            q[:] = 0  # an empty shard
        shards.append(q)
    if not any(int(q.sum()) for q in shards):
        shards[0][0] = 1
    leaves = np.concatenate(shards)
    S = int(sum(int(q.sum()) for q in shards))
    prefix = np.cumsum([0] + [int(q.sum()) for q in shards])
    offsets = np.cumsum([0] + [len(q) for q in shards])
    B, seed, rnd = int(rng.integers(1, 60)), 5 + case, case
    g_idx, g_q = orc.sample_prioritized_scan(leaves, B, seed, rnd)
    owners = []
    for k in range(B):
        t = orc.stratum_target(S, B, k, orc.philox_u64(seed, k, rnd, 1))
        owner = int(np.searchsorted(prefix, t, side="right")) - 1
        owners.append(owner)
        assert prefix[owner] <= t < prefix[owner + 1]
        local = _inverse_cdf(shards[owner], t - int(prefix[owner]))
        assert offsets[owner] + local == g_idx[k]
        assert shards[owner][local] == g_q[k]
    assert owners == sorted(owners)  # grouped by owner, stratum order kept


def _dying_rank(rank, world, port, out):
    import datetime
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    from paper_2609_24456_gb300.shard import ShardComm
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world,
                            timeout=datetime.timedelta(seconds=5))
    c = ShardComm()
    c.all_gather(torch.tensor([rank]))  # one exchange that both ranks make
    if rank == 1:
        os._exit(0)  # leaves between exchanges, without a word
    try:
        c.all_gather(torch.tensor([rank]))  # the next round's first exchange
        out.put("no error")
    except Exception as e:  # the peer's departure surfaces here
        out.put("error: %s" % type(e).__name__)


@pytest.mark.timeout(120)
def test_a_rank_that_leaves_between_rounds_is_detected():
    """A rank that exits between two rounds (no kernel or collective of
    its own in flight) makes the other rank's next exchange fail with an
    error instead of waiting forever: the process group's timeout bounds
    it.  Host-side failure detection for the sharded buffer."""
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_dying_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = q.get(timeout=100)
    for p in procs:
        p.join(timeout=30)
    assert res.startswith("error"), res
