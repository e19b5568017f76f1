"""Online placement migration (edp_migrate) through the C ABI.

A ring's state moves into an empty context with another placement: the
multimodal two-tier ring into single-tier, wider, narrower, larger and
smaller rings, and a prioritized frame-stack ring into a larger one.  The
destination receives the source's newest n transitions as its first n
insertions.  After the move it must behave exactly as a ring that had
received those transitions from the start: every one in the tier and slot
the placement map gives, deliveries bit-exact against the oracle, the
priority tree (leaves, every internal sum, deferred and maximum priority)
equal to the oracle's -- and it must keep working after further
insertions.  The source is left unchanged.
"""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, check_tree, dqn_outputs, fx, to_np, u32
from test_gpu_mm import Logical, _deliver_check, _ingest, _mm_ring

pytestmark = pytest.mark.gpu

INGESTS = [30, 20, 64, 1, 50, 24, 25]  # 214 transitions in all


def _renumbered(lg, dst_cap):
    """The oracle of the destination: the source's newest n transitions as
    insertions 0 .. n-1 of a ring of dst_cap slots."""
    n = min(lg.total, lg.cap, dst_cap)
    L0 = lg.total - n
    ref = Logical(dst_cap, lg.seed)
    for j in range(n):
        ref.obs[j % dst_cap] = lg.obs[(L0 + j) % lg.cap]
        ref.tok[j % dst_cap] = lg.tok[(L0 + j) % lg.cap]
        ref.rew[j % dst_cap] = lg.rew[(L0 + j) % lg.cap]
    ref.total = n
    return ref


@pytest.mark.parametrize("dst_cap,dst_cap_h", [(64, 64), (64, 40), (100, 30), (40, 10),
                                               (300, 300)])
def test_migrate_two_tier_ring(edp_lib, orc, dst_cap, dst_cap_h):
    edp = edp_lib
    src_cap, src_cap_h, seed = 64, 24, 6
    src = _mm_ring(edp, src_cap, src_cap_h)
    lg = Logical(src_cap, seed)
    for n in INGESTS:
        _ingest(edp, src, lg, orc, n, seed)
    dst = _mm_ring(edp, dst_cap, dst_cap_h)
    edp.edp_migrate(src.ctx, dst.ctx)
    edp.edp_sync(dst.ctx)
    ref = _renumbered(lg, dst_cap)
    assert dst.info().total == ref.total
    # placement: each transition where the destination's map puts it
    host = dst.host_obs.numpy() if dst.host_obs is not None else None
    hbm = dst.obs.cpu().numpy()
    for j in range(ref.total):
        tier, slot = orc.tier_of(dst_cap, dst_cap_h, ref.total, j)
        row = host[slot] if tier == 1 else hbm[slot]
        assert np.array_equal(row, ref.obs[j % dst_cap]), (j, tier)
    for rnd in range(3):
        _deliver_check(edp, orc, dst, ref, 48, seed=11, rnd=rnd)
    # the source is unchanged and still delivers
    _deliver_check(edp, orc, src, lg, 48, seed=11, rnd=7)
    # the destination keeps working: more insertions after the move
    _ingest(edp, dst, ref, orc, 17, seed)
    _deliver_check(edp, orc, dst, ref, 48, seed=12, rnd=0)


def test_migrate_prioritized_frame_stack(edp_lib, orc):
    edp = edp_lib
    Fb = 84 * 16
    frames, action, reward, done = fx.dqn_transitions(50, 2700, Fb, done_p=0.05)
    q = orc.priorities_from_td(fx.td_errors(50, 2700), 0.6, 1e-6)
    src = MirroredDqn(1000, prioritized=True, F=Fb)
    t = 0
    for n in [700, 900, 1000]:
        sl = slice(t, t + n)
        src.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
        t += n
    dst = MirroredDqn(3000, prioritized=True, F=Fb)
    edp.edp_migrate(src.ring.ctx, dst.ring.ctx)
    edp.edp_sync(dst.ring.ctx)
    # oracle of the destination: the source's 1,000 retained transitions as
    # its first 1,000 insertions
    L0 = t - 1000
    js = np.arange(1000)
    srcs = (L0 + js) % 1000
    dst.frames[js] = src.frames[srcs]
    dst.action[js] = src.action[srcs]
    dst.reward[js] = src.reward[srcs]
    dst.done[js] = src.done[srcs]
    dst.st.leaves[js] = src.st.leaves[srcs]
    dst.st.pending[:] = src.st.pending
    dst.st.qmax[:] = src.st.qmax
    dst.total = 1000
    check_tree(orc, dst.ring, dst.st)

    def round_check(seed, rnd):
        B = 256
        idx = torch.empty(B, dtype=torch.int64, device="cuda")
        qs = torch.empty(B, dtype=torch.int32, device="cuda")
        edp.edp_sample(dst.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, B, seed, rnd, idx, qs)
        obs, nxt, act, rew, dn = dqn_outputs(B, 4, Fb)
        edp.edp_deliver(dst.ring.ctx, idx, B, edp.make_batch(obs, nxt, act, rew, dn))
        edp.edp_sync(dst.ring.ctx)
        ref_idx, ref_q = orc.sample_prioritized_bisect(dst.st.leaves, B, seed, rnd)
        assert np.array_equal(to_np(idx), ref_idx)
        assert np.array_equal(u32(qs), ref_q)
        r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
            dst.frames, dst.done, dst.action, dst.reward, dst.cap, dst.total, 4, ref_idx)
        assert np.array_equal(bits(obs).reshape(r_obs.shape), r_obs.view(np.uint32))
        assert np.array_equal(bits(nxt).reshape(r_nxt.shape), r_nxt.view(np.uint32))
        assert np.array_equal(to_np(act), r_act)
        assert np.array_equal(bits(rew), r_rew.view(np.uint32))
        assert np.array_equal(to_np(dn), r_dn)

    round_check(5, 1)
    # more insertions into the destination: the deferred leaf resolves
    sl = slice(t, t + 100)
    dst.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
    edp.edp_sync(dst.ring.ctx)
    check_tree(orc, dst.ring, dst.st)
    round_check(6, 2)


def test_migrate_rejects_mismatch(edp_lib, orc):
    edp = edp_lib
    a = _mm_ring(edp, 64, 24)
    b = MirroredDqn(64)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_migrate(a.ctx, b.ring.ctx)
    assert e.value.status == edp.EDP_ERR_STATE
    c = _mm_ring(edp, 64, 24)
    _ingest(edp, c, Logical(64, 1), orc, 5, 1)
    with pytest.raises(edp.EdpError) as e:  # destination not empty
        edp.edp_migrate(a.ctx, c.ctx)
    assert e.value.status == edp.EDP_ERR_STATE
