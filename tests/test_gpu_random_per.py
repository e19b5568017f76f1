"""Randomised prioritized-replay rounds against the oracle: rings of 40 to
40,000 slots filled past a wrap in random chunks with random priorities
(some zero, some at the running maximum), frame stacks of 1 to 8 with and
without next_obs, batches of 1 to 2,000 on both sides of the staged
delivery's threshold; per round the indices, priorities and whole batch
bit-exact, IS weights within 1 ulp, then a priority update (u32 or from TD
errors, with repeats, the deferred newest transition and slots that hold
nothing) after which every node of the tree is compared."""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, check_tree, cuda, dqn_outputs, fx, to_np, u32

pytestmark = pytest.mark.gpu

ALPHA, EPS = 0.6, 1e-6


def _ulps(a, b):
    return np.abs(a.view(np.int32).astype(np.int64) - b.view(np.int32).astype(np.int64))


@pytest.mark.parametrize("seed", range(16))
def test_random_prioritized_rounds(edp_lib, orc, seed):
    edp = edp_lib
    rng = np.random.default_rng(11000 + seed)
    cap = int(rng.choice([int(rng.integers(40, 400)), int(rng.integers(400, 40000))]))
    K = int(rng.integers(1, 9))
    nxt = bool(rng.integers(0, 2))
    F = 84 * 4
    m = MirroredDqn(cap, K=K, next_obs=nxt, prioritized=True, F=F)
    total_n = int(cap * rng.uniform(0.6, 2.2)) + 3
    frames, action, reward, done = fx.dqn_transitions(11000 + seed, total_n, F,
                                                      done_p=float(rng.choice([0.0, 0.02, 0.2])))
    q = orc.priorities_from_td(fx.td_errors(11000 + seed, total_n), ALPHA, EPS)
    q[rng.random(total_n) < 0.1] = 0
    t = 0
    while t < total_n:
        n = int(min(total_n - t, rng.integers(1, cap + 1)))
        sl = slice(t, t + n)
        default = rng.random() < 0.2  # leaves at the running maximum
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=None if default else q[sl])
        t += n
    beta = float(rng.uniform(0.2, 1.0))
    for rnd in range(3):
        if int(m.st.leaves.astype(np.uint64).sum()) == 0:
            break
        B = int(rng.choice([int(rng.integers(1, 64)), int(rng.integers(64, 2001))]))
        s = int(rng.integers(0, 1 << 30))
        idx = torch.full((B,), -5, dtype=torch.int64, device="cuda")
        qs = torch.zeros(B, dtype=torch.int32, device="cuda")
        edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, B, s, rnd, idx, qs)
        obs, nx, act, rew, dn = dqn_outputs(B, K, F, with_next=nxt)
        isw = torch.full((B,), float("nan"), device="cuda")
        edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(obs, nx, act, rew, dn, q=qs,
                                                           isw=isw, beta=beta))
        edp.edp_sync(m.ring.ctx)
        ref_idx, ref_q = orc.sample_prioritized_bisect(m.st.leaves, B, s, rnd)
        assert np.array_equal(to_np(idx), ref_idx), (seed, rnd)
        assert np.array_equal(u32(qs), ref_q)
        assert _ulps(to_np(isw), orc.is_weights(ref_q, beta)).max() <= 1
        r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
            m.frames, m.done, m.action, m.reward, cap, m.total, K, ref_idx, with_next=nxt)
        assert np.array_equal(bits(obs).reshape(r_obs.shape), r_obs.view(np.uint32))
        if nxt:
            assert np.array_equal(bits(nx).reshape(r_nxt.shape), r_nxt.view(np.uint32))
        assert np.array_equal(to_np(act), r_act) and np.array_equal(to_np(dn), r_dn)
        assert np.array_equal(bits(rew), r_rew.view(np.uint32))
        # the update: the sampled slots, repeats, the newest slot and slots
        # that hold nothing (when the ring is not full)
        n_up = int(rng.integers(1, 3000))
        up = rng.choice(ref_idx, size=n_up).astype(np.int64)
        up[rng.random(n_up) < 0.05] = int((m.total - 1) % cap)
        up[rng.random(n_up) < 0.05] = int(rng.integers(0, cap))
        if rng.integers(0, 2):
            d_td = cuda((rng.standard_normal(n_up) * 2).astype(np.float32))
            qd = torch.zeros(n_up, dtype=torch.int32, device="cuda")
            edp.edp_priorities_from_td(m.ring.ctx, d_td, n_up, ALPHA, EPS, qd)
            edp.edp_update_priorities_td(m.ring.ctx, cuda(up), d_td, n_up, ALPHA, EPS)
            edp.edp_sync(m.ring.ctx)
            qu = u32(qd)
        else:
            qu = rng.integers(0, 1 << 31, size=n_up).astype(np.uint32)
            edp.edp_update_priorities(m.ring.ctx, cuda(up), cuda(qu.view(np.int32)), n_up)
        orc.update_leaves(m.st, m.total, up, qu)
        edp.edp_sync(m.ring.ctx)
        check_tree(orc, m.ring, m.st)
    m.ring.close()
