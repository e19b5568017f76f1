"""GPU parity of prioritized replay through the C ABI: the fixed-point
sum-tree (every node bit-exact), stratified sampling (indices and
priorities bit-exact), IS weights (within 1 ulp), priority updates with
duplicates and the deferred newest priority, at small sizes and at the
1,000,000-frame replay size."""
import numpy as np
import pytest
import torch

from gpu_util import (MirroredDqn, bits, check_tree, cuda, dqn_outputs, fx,
                      to_np, u32)

pytestmark = pytest.mark.gpu

ALPHA, EPS, BETA = 0.6, 1e-6, 0.4


def _ulp_diff(a, b):
    a = a.view(np.int32).astype(np.int64)
    b = b.view(np.int32).astype(np.int64)
    return np.abs(a - b)


def _round(edp, orc, m, B, seed, rnd, td_seed, check_outputs=True, subset=None):
    ctx = m.ring.ctx
    idx = torch.full((B,), -5, dtype=torch.int64, device="cuda")
    q = torch.zeros(B, dtype=torch.int32, device="cuda")
    edp.edp_sample(ctx, edp.EDP_SAMPLE_PRIORITIZED, B, seed, rnd, idx, q)
    obs, nxt, act, rew, dn = dqn_outputs(B, m.K, m.F)
    isw = torch.full((B,), float("nan"), dtype=torch.float32, device="cuda")
    edp.edp_deliver(ctx, idx, B, edp.make_batch(obs, nxt, act, rew, dn, q=q,
                                                isw=isw, beta=BETA))
    edp.edp_sync(ctx)
    ref_idx, ref_q = orc.sample_prioritized_bisect(m.st.leaves, B, seed, rnd)
    assert np.array_equal(to_np(idx), ref_idx)
    assert np.array_equal(u32(q), ref_q)
    ref_w = orc.is_weights(ref_q, BETA)
    assert _ulp_diff(to_np(isw), ref_w).max() <= 1
    if check_outputs:
        sel = np.arange(B) if subset is None else subset
        r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
            m.frames, m.done, m.action, m.reward, m.cap, m.total, m.K,
            ref_idx[sel])
        assert np.array_equal(bits(obs)[sel].reshape(r_obs.shape),
                              r_obs.view(np.uint32))
        assert np.array_equal(bits(nxt)[sel].reshape(r_nxt.shape),
                              r_nxt.view(np.uint32))
        assert np.array_equal(to_np(act)[sel], r_act)
        assert np.array_equal(bits(rew)[sel], r_rew.view(np.uint32))
        assert np.array_equal(to_np(dn)[sel], r_dn)
    # priority callback from fresh TD errors (bit-exact u32 path)
    td = fx.td_errors(td_seed, B, rnd)
    qn = orc.priorities_from_td(td, ALPHA, EPS)
    edp.edp_update_priorities(ctx, idx, cuda(qn), B)
    orc.update_leaves(m.st, m.total, ref_idx, qn)
    edp.edp_sync(ctx)
    return ref_idx


def test_tree_build_and_sampling_small(edp_lib, orc):
    edp = edp_lib
    cap = 3000  # not a power of 32: padded leaves
    N = 7000
    frames, action, reward, done = fx.dqn_transitions(1, N, done_p=0.02)
    td = fx.td_errors(1, N)
    q = orc.priorities_from_td(td, ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True)
    t = 0
    for k, n in enumerate([1, 2, 1500, 1497, 2999, 1001]):
        sl = slice(t, t + n)
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
        t += n
        edp.edp_sync(m.ring.ctx)
        check_tree(orc, m.ring, m.st)
        if m.total >= 2:
            _round(edp, orc, m, 100 + k, seed=11, rnd=k, td_seed=100 + k)
            check_tree(orc, m.ring, m.st)


def test_update_duplicates_invalid_and_deferred(edp_lib, orc):
    edp = edp_lib
    cap = 500
    frames, action, reward, done = fx.dqn_transitions(2, 800)
    q = orc.priorities_from_td(fx.td_errors(2, 800), ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True)
    m.ingest(orc, frames[:300], action[:300], reward[:300], done[:300], q=q[:300])
    rng = np.random.default_rng(3)
    for step in range(6):
        n = 5000 + step  # several 4096-pair chunks, many duplicates
        idx = rng.integers(0, 320, size=n).astype(np.int64)
        idx[::7] = idx[0]
        idx[5] = m.total - 1  # the newest (deferred) transition
        qu = rng.integers(0, 1 << 31, size=n).astype(np.uint32)
        edp.edp_update_priorities(m.ring.ctx, cuda(idx), cuda(qu), n)
        orc.update_leaves(m.st, m.total, idx, qu)
        edp.edp_sync(m.ring.ctx)
        check_tree(orc, m.ring, m.st)
    # an index outside [0, cap) is skipped on the device and reported
    bad = np.array([3, -1, 7, cap + 5], np.int64)
    qb = np.array([10, 20, 30, 40], np.uint32)
    edp.edp_update_priorities(m.ring.ctx, cuda(bad), cuda(qb), 4)
    orc.update_leaves(m.st, m.total, bad, qb)
    status, msg = edp.edp_sync_status(m.ring.ctx)
    assert status == edp.EDP_ERR_INVALID, msg
    check_tree(orc, m.ring, m.st)
    # the deferred priority lands when the successor arrives
    m.ingest(orc, frames[300:301], action[300:301], reward[300:301],
             done[300:301], q=q[300:301])
    edp.edp_sync(m.ring.ctx)
    check_tree(orc, m.ring, m.st)
    # default priority (running maximum) for q == NULL
    m.ingest(orc, frames[301:310], action[301:310], reward[301:310], done[301:310])
    edp.edp_sync(m.ring.ctx)
    check_tree(orc, m.ring, m.st)


@pytest.mark.parametrize("n", [1, 31, 33, 512, 2048, 2049, 5000])
@pytest.mark.parametrize("path", ["u32", "td"])
def test_update_batch_sizes(edp_lib, orc, n, path):
    """Both entry points at batch sizes from one pair to several of the
    update's 1,024-pair chunks: duplicates (last wins), the deferred newest
    transition, slots outside the stored range, then the whole tree
    bit-exact.  The TD-error path is checked against the oracle
    applying the priorities the device's own rule gives for the same TD
    errors (edp_priorities_from_td), so the tree comparison stays exact."""
    edp = edp_lib
    cap = 3000
    frames, action, reward, done = fx.dqn_transitions(11, 2500, 84 * 4)
    q = orc.priorities_from_td(fx.td_errors(11, 2500), ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True, F=84 * 4)
    m.ingest(orc, frames, action, reward, done, q=q)
    rng = np.random.default_rng(n * 3 + (path == "td"))
    for step in range(3):
        idx = rng.integers(0, 2600, size=n).astype(np.int64)  # 2500.. hold nothing
        idx[::7] = idx[0]
        if n > 5:
            idx[5] = m.total - 1  # the newest (deferred) transition
        if path == "u32":
            qu = rng.integers(0, 1 << 31, size=n).astype(np.uint32)
            edp.edp_update_priorities(m.ring.ctx, cuda(idx), cuda(qu), n)
        else:
            td = rng.standard_normal(n).astype(np.float32) * 3
            d_td = cuda(td)
            qd = torch.zeros(n, dtype=torch.int32, device="cuda")
            edp.edp_priorities_from_td(m.ring.ctx, d_td, n, ALPHA, EPS, qd)
            edp.edp_update_priorities_td(m.ring.ctx, cuda(idx), d_td, n, ALPHA, EPS)
            edp.edp_sync(m.ring.ctx)
            qu = u32(qd)
        orc.update_leaves(m.st, m.total, idx, qu)
        edp.edp_sync(m.ring.ctx)
        check_tree(orc, m.ring, m.st)


@pytest.mark.parametrize("cap", [20, 33, 500])
@pytest.mark.parametrize("path", ["u32", "td"])
def test_update_shallow_trees(edp_lib, orc, cap, path):
    """Trees of depth 1 (20 leaves under the root), 2 (33 and 500 leaves):
    the single-pass update's level-1 and root sums on their own, batches of
    1 to 300 pairs with repeats, slots that hold nothing and the deferred
    newest transition; the whole tree bit-exact after each."""
    edp = edp_lib
    n_in = cap - 3
    frames, action, reward, done = fx.dqn_transitions(23, n_in, 84 * 4)
    q0 = orc.priorities_from_td(fx.td_errors(23, n_in), ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True, F=84 * 4)
    m.ingest(orc, frames, action, reward, done, q=q0)
    rng = np.random.default_rng(cap * 7 + (path == "td"))
    for n in (1, 7, 40, 300):
        idx = rng.integers(0, cap, size=n).astype(np.int64)  # cap - 3 .. hold nothing
        idx[n // 2] = m.total - 1
        if path == "u32":
            qu = rng.integers(0, 1 << 31, size=n).astype(np.uint32)
            edp.edp_update_priorities(m.ring.ctx, cuda(idx), cuda(qu), n)
        else:
            d_td = cuda((rng.standard_normal(n) * 3).astype(np.float32))
            qd = torch.zeros(n, dtype=torch.int32, device="cuda")
            edp.edp_priorities_from_td(m.ring.ctx, d_td, n, ALPHA, EPS, qd)
            edp.edp_update_priorities_td(m.ring.ctx, cuda(idx), d_td, n, ALPHA, EPS)
            edp.edp_sync(m.ring.ctx)
            qu = u32(qd)
        orc.update_leaves(m.st, m.total, idx, qu)
        edp.edp_sync(m.ring.ctx)
        check_tree(orc, m.ring, m.st)


def test_small_updates_queued_back_to_back(edp_lib, orc):
    """Single-pass updates (up to 2,048 pairs) queued straight after each
    other on one stream, with nothing between them: each waits for the one
    before, so the later batch wins on the slots both touch.  Four calls
    (TD errors and u32 priorities, 2,048 / 513 / 32 / 1 pairs, many shared
    slots and the deferred newest one), then the whole tree bit-exact."""
    edp = edp_lib
    cap = 3000
    frames, action, reward, done = fx.dqn_transitions(17, 2600, 84 * 4)
    q0 = orc.priorities_from_td(fx.td_errors(17, 2600), ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True, F=84 * 4)
    m.ingest(orc, frames, action, reward, done, q=q0)
    rng = np.random.default_rng(18)
    calls = []
    for k, n in enumerate((2048, 513, 32, 1)):
        idx = rng.integers(0, 300, size=n).astype(np.int64)  # shared slots
        idx[n // 2] = m.total - 1  # the newest (deferred) transition
        if k % 2 == 0:
            td = (rng.standard_normal(n) * 2).astype(np.float32)
            d_td = cuda(td)
            qd = torch.zeros(n, dtype=torch.int32, device="cuda")
            edp.edp_priorities_from_td(m.ring.ctx, d_td, n, ALPHA, EPS, qd)
            calls.append((cuda(idx), d_td, None, n, idx, qd))
        else:
            qu = rng.integers(1, 1 << 31, size=n).astype(np.uint32)
            calls.append((cuda(idx), None, cuda(qu.view(np.int32)), n, idx, qu))
    torch.cuda.synchronize()
    for d_idx, d_td, d_q, n, _, _ in calls:
        if d_td is not None:
            edp.edp_update_priorities_td(m.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
        else:
            edp.edp_update_priorities(m.ring.ctx, d_idx, d_q, n)
    edp.edp_sync(m.ring.ctx)
    for _, _, _, _, idx, q in calls:
        orc.update_leaves(m.st, m.total, idx, u32(q) if torch.is_tensor(q) else q)
    check_tree(orc, m.ring, m.st)


def test_priorities_from_td_within_one(edp_lib, orc):
    edp = edp_lib
    m = MirroredDqn(64, prioritized=True)
    td = fx.td_errors(5, 1 << 20)
    td[:4] = [0.0, -3.0, 1e-30, 1e6]
    q = torch.zeros(len(td), dtype=torch.int32, device="cuda")
    edp.edp_priorities_from_td(m.ring.ctx, cuda(td), len(td), ALPHA, EPS, q)
    edp.edp_sync(m.ring.ctx)
    ref = orc.priorities_from_td(td, ALPHA, EPS).astype(np.int64)
    diff = np.abs(u32(q).astype(np.int64) - ref)
    assert diff.max() <= 1
    assert (diff > 0).mean() < 1e-3
    # the ends of the clamp are exact: a zero error without eps, and errors
    # whose priority exceeds 32 bits
    ends = np.array([0.0, 1e9, -1e9, 0.0], np.float32)
    qe = torch.zeros(4, dtype=torch.int32, device="cuda")
    edp.edp_priorities_from_td(m.ring.ctx, cuda(ends), 4, ALPHA, 0.0, qe)
    edp.edp_sync(m.ring.ctx)
    assert u32(qe).tolist() == orc.priorities_from_td(ends, ALPHA, 0.0).tolist()
    assert u32(qe).tolist() == [1, 2**32 - 1, 2**32 - 1, 1]


@pytest.mark.parametrize("alpha,eps", [(1.0, 0.0), (0.05, 1e-6), (0.4, 1e-2),
                                       (1.5, 1e-6), (0.0, 1e-6)])
def test_priorities_from_td_other_exponents(edp_lib, orc, alpha, eps):
    """The rule at other exponents and offsets: (0, 1] takes the
    double-float evaluation, 0 and exponents above 1 the fp64 one; errors
    from 1e-30 to 3e38 (beyond 2^100 the fp64 one again).  Within one of
    the oracle, and rarely off by one (an exponent of 1 with no offset
    makes exact ties, which a rounding step may resolve either way)."""
    edp = edp_lib
    m = MirroredDqn(64, prioritized=True)
    rng = np.random.default_rng(int(alpha * 100) + int(eps * 1e6))
    td = np.exp(rng.uniform(np.log(1e-30), np.log(3e38), 1 << 18)).astype(np.float32)
    td[: 1 << 17] = fx.td_errors(6, 1 << 17)
    td *= np.where(rng.random(len(td)) < 0.5, -1, 1).astype(np.float32)
    q = torch.zeros(len(td), dtype=torch.int32, device="cuda")
    edp.edp_priorities_from_td(m.ring.ctx, cuda(td), len(td), alpha, eps, q)
    edp.edp_sync(m.ring.ctx)
    ref = orc.priorities_from_td(td, alpha, eps).astype(np.int64)
    diff = np.abs(u32(q).astype(np.int64) - ref)
    assert diff.max() <= 1
    assert (diff > 0).mean() < 1e-3


def test_all_zero_priorities_report_empty(edp_lib, orc):
    edp = edp_lib
    m = MirroredDqn(40, prioritized=True)
    frames, action, reward, done = fx.dqn_transitions(4, 20)
    m.ingest(orc, frames, action, reward, done, q=np.zeros(20, np.uint32))
    idx = torch.zeros(8, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, 8, 0, 0, idx)
    status, msg = edp.edp_sync_status(m.ring.ctx)
    assert status == edp.EDP_ERR_EMPTY, msg
    assert (to_np(idx) == -1).all()


def test_prioritized_replay_full_size(edp_lib, orc):
    """1,000,000 uint8 84x84 frames (~7 GB) with PER priorities from Exp(1)
    TD errors; batch 512; three sample/deliver/update rounds.  Indices,
    priorities and the whole tree are compared in full; delivered stacks on
    a subset of the batch (the oracle reads only the frames it needs)."""
    edp = edp_lib
    cap, F, B = 1_000_000, 84 * 84, 512
    seed = 1235
    m = MirroredDqn(cap, prioritized=True)
    # metadata from the numpy fixtures; frames from the content function
    _, action, reward, done = fx.dqn_transitions(seed, cap, with_frames=False)
    q = orc.priorities_from_td(fx.td_errors(seed, cap), ALPHA, EPS)
    chunk = 65536
    staging = torch.empty((chunk, F), dtype=torch.uint8, device="cuda")
    for lo in range(0, cap, chunk):
        hi = min(cap, lo + chunk)
        n = hi - lo
        fx.content_fill_torch(seed, lo, staging[:n])
        edp.edp_ingest(m.ring.ctx, staging[:n], n, action=cuda(action[lo:hi]),
                       reward=cuda(reward[lo:hi]), done=cuda(done[lo:hi]),
                       q=cuda(q[lo:hi]))
        orc.ingest_leaves(m.st, lo, q[lo:hi])
    m.total = cap
    m.action, m.reward, m.done = action, reward, done
    # sparse oracle frame store: only the frames the checked subset needs
    m.frames = np.zeros((cap, F), np.uint8)
    edp.edp_sync(m.ring.ctx)
    check_tree(orc, m.ring, m.st)
    subset = np.arange(0, B, 37)
    for rnd in range(3):
        ref_idx, _ = orc.sample_prioritized_bisect(m.st.leaves, B, 7, rnd)
        need = set()
        for s in ref_idx[subset]:
            for o in range(-3, 2):
                need.add((int(s) + o) % cap)
        need = sorted(need)
        m.frames[need] = fx.content_bytes(seed, need, F)  # id == slot here
        _round(edp, orc, m, B, seed=7, rnd=rnd, td_seed=900 + rnd, subset=subset)
        check_tree(orc, m.ring, m.st)


@pytest.mark.parametrize("path", ["u32", "td"])
def test_updates_back_to_back_on_one_stream(edp_lib, orc, path):
    """Two priority updates queued straight after each other on one stream,
    with no synchronisation (and no other work) between them, over
    overlapping slots.  The second launch may start while the first is
    still applying its pairs, so neither may touch memory the other uses
    before its wait on the preceding kernel.  Whole tree bit-exact against
    the oracle applying both batches in order (for the TD-error path, with
    the priorities the device's rule gives for the same TD errors)."""
    edp = edp_lib
    cap, n = 3000, 5000
    frames, action, reward, done = fx.dqn_transitions(12, 2500, 84 * 4)
    q = orc.priorities_from_td(fx.td_errors(12, 2500), ALPHA, EPS)
    m = MirroredDqn(cap, prioritized=True, F=84 * 4)
    m.ingest(orc, frames, action, reward, done, q=q)
    rng = np.random.default_rng(41 + (path == "td"))
    batches = []
    for call in range(2):
        idx = rng.integers(0, 2500, size=n).astype(np.int64)
        idx[: n // 2] = rng.integers(0, 500, size=n // 2)  # slots both batches hit
        idx[7] = m.total - 1  # the newest (deferred) transition
        if path == "u32":
            qu = rng.integers(0, 1 << 31, size=n).astype(np.uint32)
            batches.append((cuda(idx), cuda(qu), idx, qu))
        else:
            td = (rng.standard_normal(n) * 3).astype(np.float32)
            d_td = cuda(td)
            qd = torch.zeros(n, dtype=torch.int32, device="cuda")
            edp.edp_priorities_from_td(m.ring.ctx, d_td, n, ALPHA, EPS, qd)
            edp.edp_sync(m.ring.ctx)
            batches.append((cuda(idx), d_td, idx, u32(qd)))
    torch.cuda.synchronize()
    for d_idx, d_val, _, _ in batches:  # back to back, nothing between
        if path == "u32":
            edp.edp_update_priorities(m.ring.ctx, d_idx, d_val, n)
        else:
            edp.edp_update_priorities_td(m.ring.ctx, d_idx, d_val, n, ALPHA, EPS)
    edp.edp_sync(m.ring.ctx)
    for _, _, idx, qu in batches:
        orc.update_leaves(m.st, m.total, idx, qu)
    check_tree(orc, m.ring, m.st)
