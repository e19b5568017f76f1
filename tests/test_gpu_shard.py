"""The sharded buffer (Sec. 5.1's shared-GPU placement) against the oracle's
single global buffer.

Ranks run as separate processes that share the one GPU, each with its own
shard (an edp context) and learner, exchanging through gloo with the
collectives staged in host memory (paper_2609_24456_gb300.shard.ShardComm).
No kernel of one rank waits on another's: every exchange happens on the host
between kernel launches.

Prioritized replay, G = 1, 2 and 3 shards: each shard ingests its own
transitions (its own episodes, priorities and a wrap of its ring); every
round each learner samples its strata of the global batch, gets its rows,
and sends priority updates back (u32 priorities on even rounds, TD errors on
odd ones).  The oracle samples the concatenation of all shards' leaves
(shard-major) with the same seed and round: every learner's slots, owners
and priorities must equal the oracle's, bit for bit; importance weights
within 1 ulp of the oracle's over the whole global batch; the rows equal the
oracle's delivery from the owning shard's ring; after the rounds every
shard's tree equals the oracle's leaves after the same updates in global
batch order.

On-policy GAE with environments split over 2 ranks: the advantages, returns
and globally normalised advantages within 1e-5 of the oracle's over all
environments.
"""
import os
import socket
import sys
import tempfile

import numpy as np
import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CAP, N_INGEST, BL, ROUNDS, SEED = 2000, 2300, 96, 5, 31
ALPHA, EPS, BETA = 0.6, 1e-6, 0.4


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _inputs(orc, rank):
    """Fixture transitions and priorities of shard `rank`."""
    from paper_2609_24456_gb300 import fixtures as fx
    frames, action, reward, done = fx.dqn_transitions(60 + rank, N_INGEST, done_p=0.04)
    q = orc.priorities_from_td(fx.td_errors(60 + rank, N_INGEST), ALPHA, EPS)
    return frames, action, reward, done, q


def _update_values(orc, rank, r):
    """This learner's TD errors of round r and the priorities they give."""
    from paper_2609_24456_gb300 import fixtures as fx
    td = fx.td_errors(90 + rank, BL, r)
    return td, orc.priorities_from_td(td, ALPHA, EPS)


def _per_rank(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch
    import torch.distributed as dist
    import oracle as orc
    from gpu_util import MirroredDqn, cuda, tree_levels, to_np, bits
    from paper_2609_24456_gb300 import edp
    from paper_2609_24456_gb300.shard import ShardComm, ShardedPer
    torch.cuda.set_device(0)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        m = MirroredDqn(CAP, prioritized=True)
        frames, action, reward, done, q = _inputs(orc, rank)
        half = N_INGEST // 2
        for sl in (slice(0, half), slice(half, N_INGEST)):  # the second wraps
            m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
        sp = ShardedPer(m.ring, ShardComm(), BL, beta=BETA, alpha=ALPHA, eps=EPS)
        res = {}
        for r in range(ROUNDS):
            lo, owner = sp.sample_deliver(SEED, r)
            torch.cuda.synchronize()
            for k in ("obs", "nxt", "rew", "isw"):
                res["%s_%d" % (k, r)] = bits(lo[k])
            for k in ("act", "done", "idx"):
                res["%s_%d" % (k, r)] = to_np(lo[k])
            res["q_%d" % r] = to_np(lo["q"]).view(np.uint32)
            res["owner_%d" % r] = owner.numpy()
            td, qu = _update_values(orc, rank, r)
            if r % 2 == 0:
                sp.update(q=cuda(qu))
            else:
                sp.update(td=cuda(td))
        edp.edp_sync(m.ring.ctx)
        leaves, lv, pending, qmax = tree_levels(m.ring)
        res["leaves"] = leaves[:CAP]
        res["root"] = np.array([lv[0][0]], np.uint64)
        np.savez(os.path.join(out_dir, "per_%d.npz" % rank), **res)
    finally:
        dist.destroy_process_group()


def _gae_rank(rank, world, port, out_dir):
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import torch
    import torch.distributed as dist
    from gpu_util import cuda, to_np
    from paper_2609_24456_gb300 import edp
    from paper_2609_24456_gb300 import fixtures as fx
    from paper_2609_24456_gb300.shard import ShardComm, sharded_gae
    torch.cuda.set_device(0)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        T, E = 64, 96
        _, r, v, d = fx.ppo_rollout(7, T, E, done_p=0.02, with_obs=False)
        El = E // world
        cols = slice(rank * El, (rank + 1) * El)
        cfg = edp.make_config(16, (3, 4, 4), edp.EDP_XFORM_HWC_CHW_BF16)
        ring = edp.Ring(cfg, action=False, reward=False, done=False)
        adv = torch.empty((T, El), device="cuda")
        ret = torch.empty((T, El), device="cuda")
        nrm = torch.empty((T, El), device="cuda")
        stats = torch.zeros(3, dtype=torch.float64, device="cuda")
        sharded_gae(ring.ctx, ShardComm(), cuda(np.ascontiguousarray(r[:, cols])),
                    cuda(np.ascontiguousarray(v[:, cols])),
                    cuda(np.ascontiguousarray(d[:, cols])), T, El, 0.99, 0.95, adv, ret,
                    nrm, stats)
        edp.edp_sync(ring.ctx)
        np.savez(os.path.join(out_dir, "gae_%d.npz" % rank), adv=to_np(adv), ret=to_np(ret),
                 nrm=to_np(nrm), stats=to_np(stats))
        ring.close()
    finally:
        dist.destroy_process_group()


def _spawn(fn, world, out_dir):
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    port = _free_port()
    procs = [ctx.Process(target=fn, args=(r, world, port, out_dir)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=240)
    for p in procs:
        if p.is_alive():
            p.kill()
        assert p.exitcode == 0, "rank process failed (exit %s)" % p.exitcode


def _ulps(a, b):
    a = np.asarray(a, np.float32).view(np.int32).astype(np.int64)
    b = np.asarray(b, np.float32).view(np.int32).astype(np.int64)
    return int(np.abs(a - b).max()) if a.size else 0


@pytest.mark.timeout(600)
@pytest.mark.parametrize("world", [1, 2, 3])
def test_sharded_per_equals_one_global_buffer(orc, world):
    with tempfile.TemporaryDirectory() as out_dir:
        _spawn(_per_rank, world, out_dir)
        got = [dict(np.load(os.path.join(out_dir, "per_%d.npz" % g))) for g in range(world)]
    # the oracle's shards: ring arrays and leaves, fed the same inputs
    shards = []
    for g in range(world):
        frames, action, reward, done, q = _inputs(orc, g)
        ring = {"frames": np.zeros((CAP, 84 * 84), np.uint8),
                "action": np.zeros(CAP, np.int32), "reward": np.zeros(CAP, np.float32),
                "done": np.zeros(CAP, np.uint8)}
        st = orc.PerState(CAP, True)
        half = N_INGEST // 2
        total = 0
        for sl in (slice(0, half), slice(half, N_INGEST)):
            n = sl.stop - sl.start
            for key, src in (("frames", frames), ("action", action), ("reward", reward),
                             ("done", done)):
                orc.ring_write(ring[key], CAP, total, np.ascontiguousarray(src[sl]))
            orc.ingest_leaves(st, total, q[sl])
            total += n
        shards.append((ring, st, total))
    B = world * BL
    for r in range(ROUNDS):
        leaves = np.concatenate([st.leaves for _, st, _ in shards])
        g_idx, g_q = orc.sample_prioritized_bisect(leaves, B, SEED, r)
        g_w = orc.is_weights(g_q, BETA)
        upd = [[] for _ in range(world)]  # per owner: (slot, q) in global batch order
        for lr in range(world):
            sl = slice(lr * BL, (lr + 1) * BL)
            owner, slot = g_idx[sl] // CAP, g_idx[sl] % CAP
            d = got[lr]
            assert np.array_equal(d["owner_%d" % r], owner), (world, r, lr)
            assert np.array_equal(d["idx_%d" % r], slot), (world, r, lr)
            assert np.array_equal(d["q_%d" % r], g_q[sl]), (world, r, lr)
            assert _ulps(d["isw_%d" % r].view(np.float32), g_w[sl]) <= 1, (world, r, lr)
            for g in range(world):
                rows = np.nonzero(owner == g)[0]
                if not len(rows):
                    continue
                ring, st, total = shards[g]
                r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
                    ring["frames"], ring["done"], ring["action"], ring["reward"], CAP, total,
                    4, slot[rows])
                assert np.array_equal(d["obs_%d" % r][rows].reshape(r_obs.shape),
                                      r_obs.view(np.uint32)), (world, r, lr, g)
                assert np.array_equal(d["nxt_%d" % r][rows].reshape(r_nxt.shape),
                                      r_nxt.view(np.uint32)), (world, r, lr, g)
                assert np.array_equal(d["act_%d" % r][rows], r_act)
                assert np.array_equal(d["rew_%d" % r][rows], r_rew.view(np.uint32))
                assert np.array_equal(d["done_%d" % r][rows], r_dn)
            _, qu = _update_values(orc, lr, r)
            for j in range(BL):
                upd[owner[j]].append((slot[j], qu[j]))
        for g in range(world):
            if upd[g]:
                ring, st, total = shards[g]
                sl_, qs = zip(*upd[g])
                orc.update_leaves(st, total, np.array(sl_, np.int64), np.array(qs, np.uint32))
    for g in range(world):
        _, st, _ = shards[g]
        assert np.array_equal(got[g]["leaves"], st.leaves), g
        assert int(got[g]["root"][0]) == orc.leaf_sum(st.leaves, 0, CAP), g


@pytest.mark.timeout(300)
def test_sharded_gae_normalises_over_every_rank(orc):
    from paper_2609_24456_gb300 import fixtures as fx
    world, T, E = 2, 64, 96
    with tempfile.TemporaryDirectory() as out_dir:
        _spawn(_gae_rank, world, out_dir)
        got = [dict(np.load(os.path.join(out_dir, "gae_%d.npz" % g))) for g in range(world)]
    _, r, v, d = fx.ppo_rollout(7, T, E, done_p=0.02, with_obs=False)
    adv, ret = orc.gae(r, v, d, 0.99, 0.95)
    nrm = orc.normalize(adv.ravel())[0].reshape(adv.shape)
    El = E // world
    for g in range(world):
        cols = slice(g * El, (g + 1) * El)
        assert np.abs(got[g]["adv"] - adv[:, cols]).max() <= 1e-5
        assert np.abs(got[g]["ret"] - ret[:, cols]).max() <= 1e-5
        assert np.abs(got[g]["nrm"] - nrm[:, cols]).max() <= 1e-5
        assert got[g]["stats"][0] == T * E


def test_route_and_descend_one_shard_equals_prioritized_sampling(edp_lib, orc):
    """With one shard, routing over its own total and descending the local
    targets is edp_sample(PRIORITIZED): same slots and priorities; the
    given-q importance weights equal the delivery's."""
    import torch
    from gpu_util import MirroredDqn, cuda, to_np, u32
    edp = edp_lib
    m = MirroredDqn(CAP, prioritized=True)
    frames, action, reward, done, q = _inputs(orc, 0)
    half = N_INGEST // 2
    for sl in (slice(0, half), slice(half, N_INGEST)):  # the second wraps
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
    B = 300
    i64 = dict(dtype=torch.int64, device="cuda")
    total, counts = torch.zeros(1, **i64), torch.zeros(1, **i64)
    local_t, idx = torch.zeros(B, **i64), torch.zeros(B, **i64)
    qs = torch.zeros(B, dtype=torch.int32, device="cuda")
    ref_idx = torch.zeros(B, **i64)
    ref_q = torch.zeros(B, dtype=torch.int32, device="cuda")
    edp.edp_tree_total(m.ring.ctx, total)
    edp.edp_route_prioritized(m.ring.ctx, total, 1, B, 0, B, 11, 3, local_t, counts)
    edp.edp_sample_targets(m.ring.ctx, local_t, B, idx, qs)
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, B, 11, 3, ref_idx, ref_q)
    qmin = torch.zeros(1, **i64)
    w = torch.zeros(B, device="cuda")
    edp.edp_batch_qmin(m.ring.ctx, qs, B, qmin)
    edp.edp_is_weights(m.ring.ctx, qs, B, qmin, BETA, w)
    obs = torch.empty((B, 4, 84 * 84), device="cuda")
    isw = torch.empty(B, device="cuda")
    edp.edp_deliver(m.ring.ctx, ref_idx, B, edp.make_batch(obs, q=ref_q, isw=isw, beta=BETA))
    edp.edp_sync(m.ring.ctx)
    assert int(counts[0]) == B
    assert int(total[0]) == orc.leaf_sum(m.st.leaves, 0, CAP)
    assert np.array_equal(to_np(idx), to_np(ref_idx))
    assert np.array_equal(u32(qs), u32(ref_q))
    assert int(qmin[0]) == int(u32(qs).min())
    assert np.array_equal(to_np(w).view(np.uint32), to_np(isw).view(np.uint32))
    r_idx, r_q = orc.sample_prioritized_bisect(m.st.leaves, B, 11, 3)
    assert np.array_equal(to_np(idx), r_idx)


def test_sharding_calls_argument_and_device_errors(edp_lib, orc):
    import torch
    from gpu_util import MirroredDqn, cuda
    edp = edp_lib
    m = MirroredDqn(CAP, prioritized=True)
    frames, action, reward, done, q = _inputs(orc, 1)
    m.ingest(orc, frames[:500], action[:500], reward[:500], done[:500], q=q[:500])
    ctx = m.ring.ctx
    i64 = dict(dtype=torch.int64, device="cuda")
    tot, cnt = torch.zeros(4, **i64), torch.zeros(4, **i64)
    lt, idx = torch.zeros(8, **i64), torch.zeros(8, **i64)
    for G, B, k0, n in [(0, 8, 0, 8), (1025, 8, 0, 8), (1, 0, 0, 0), (1, 8, 4, 5)]:
        with pytest.raises(edp.EdpError) as e:
            edp.edp_route_prioritized(ctx, tot, G, B, k0, n, 1, 0, lt, cnt)
        assert e.value.status == edp.EDP_ERR_INVALID
    host = torch.zeros(4, dtype=torch.int64)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_route_prioritized(ctx, host, 1, 8, 0, 8, 1, 0, lt, cnt)
    assert e.value.status == edp.EDP_ERR_INVALID
    with pytest.raises(edp.EdpError) as e:
        edp.edp_is_weights(ctx, cuda(np.ones(8, np.uint32)), 8, tot, -0.5,
                           torch.zeros(8, device="cuda"))
    assert e.value.status == edp.EDP_ERR_INVALID
    # a context without priorities
    plain = MirroredDqn(64)
    for call in (lambda: edp.edp_tree_total(plain.ring.ctx, tot),
                 lambda: edp.edp_sample_targets(plain.ring.ctx, lt, 8, idx)):
        with pytest.raises(edp.EdpError) as e:
            call()
        assert e.value.status == edp.EDP_ERR_STATE
    # a target at or beyond the shard's total: idx -1, q 0, reported by sync
    edp.edp_tree_total(ctx, tot[:1])
    S = int(tot[0])
    t = cuda(np.array([0, S - 1, S, S + 5], np.uint64))
    qo = torch.full((4,), 7, dtype=torch.int32, device="cuda")
    edp.edp_sample_targets(ctx, t, 4, idx, qo)
    st, msg = edp.edp_sync_status(ctx)
    assert st == edp.EDP_ERR_INVALID, msg
    got = idx[:4].cpu().numpy()
    assert got[0] >= 0 and got[1] >= 0 and got[2] == -1 and got[3] == -1
    assert qo[2].item() == 0 and qo[3].item() == 0
    # every shard total zero: nothing routed, EDP_ERR_EMPTY at sync
    zero = torch.zeros(2, **i64)
    edp.edp_route_prioritized(ctx, zero, 2, 8, 0, 8, 1, 0, lt, cnt)
    st, msg = edp.edp_sync_status(ctx)
    assert st == edp.EDP_ERR_EMPTY, msg
    assert int(cnt[:2].sum()) == 0
