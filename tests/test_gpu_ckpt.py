"""Checkpoint / resume (edp_save, edp_load) through the C ABI.

A saved ring loaded into an empty context must behave like a ring that had
received the saved transitions, oldest first, as its first insertions: the
same oracle checks as for migration (placement by the loader's tier map,
deliveries and the whole priority tree bit-exact), for a prioritized
frame-stack ring and for a two-tier multimodal ring loaded with another
capacity and tier split; plus the error paths (foreign, truncated and
mismatched files, non-empty contexts).
"""
import numpy as np
import pytest

from gpu_util import MirroredDqn, check_tree, fx
from test_gpu_migrate import INGESTS, _renumbered
from test_gpu_mm import Logical, _deliver_check, _ingest, _mm_ring

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dst_cap,dst_cap_h", [(64, 24), (64, 64), (100, 30), (40, 10)])
def test_save_load_two_tier(edp_lib, orc, tmp_path, dst_cap, dst_cap_h):
    edp = edp_lib
    src = _mm_ring(edp, 64, 24)
    lg = Logical(64, 9)
    for n in INGESTS:
        _ingest(edp, src, lg, orc, n, 9)
    path = tmp_path / "ring.edp"
    edp.edp_save(src.ctx, str(path))
    dst = _mm_ring(edp, dst_cap, dst_cap_h)
    edp.edp_load(dst.ctx, str(path))
    edp.edp_sync(dst.ctx)
    ref = _renumbered(lg, dst_cap)
    assert dst.info().total == ref.total
    host = dst.host_obs.numpy() if dst.host_obs is not None else None
    hbm = dst.obs.cpu().numpy()
    for j in range(ref.total):
        tier, slot = orc.tier_of(dst_cap, dst_cap_h, ref.total, j)
        row = host[slot] if tier == 1 else hbm[slot]
        assert np.array_equal(row, ref.obs[j % dst_cap]), (j, tier)
    for rnd in range(3):
        _deliver_check(edp, orc, dst, ref, 48, seed=13, rnd=rnd)
    _ingest(edp, dst, ref, orc, 11, 9)  # and it keeps working
    _deliver_check(edp, orc, dst, ref, 48, seed=14, rnd=0)


def test_save_load_prioritized(edp_lib, orc, tmp_path):
    edp = edp_lib
    Fb = 84 * 16
    frames, action, reward, done = fx.dqn_transitions(70, 2700, Fb, done_p=0.05)
    q = orc.priorities_from_td(fx.td_errors(70, 2700), 0.6, 1e-6)
    src = MirroredDqn(1000, prioritized=True, F=Fb)
    t = 0
    for n in [700, 900, 1000]:
        sl = slice(t, t + n)
        src.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
        t += n
    path = tmp_path / "per.edp"
    edp.edp_save(src.ring.ctx, str(path))
    dst = MirroredDqn(1000, prioritized=True, F=Fb)
    edp.edp_load(dst.ring.ctx, str(path))
    edp.edp_sync(dst.ring.ctx)
    js = np.arange(1000)
    srcs = (t - 1000 + js) % 1000
    dst.frames[js] = src.frames[srcs]
    dst.action[js] = src.action[srcs]
    dst.reward[js] = src.reward[srcs]
    dst.done[js] = src.done[srcs]
    dst.st.leaves[js] = src.st.leaves[srcs]
    dst.st.pending[:] = src.st.pending
    dst.st.qmax[:] = src.st.qmax
    dst.total = 1000
    check_tree(orc, dst.ring, dst.st)
    sl = slice(t, t + 100)  # the deferred leaf resolves on the next insertion
    dst.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
    edp.edp_sync(dst.ring.ctx)
    check_tree(orc, dst.ring, dst.st)


def test_load_errors(edp_lib, orc, tmp_path):
    edp = edp_lib
    src = _mm_ring(edp, 64, 24)
    lg = Logical(64, 3)
    _ingest(edp, src, lg, orc, 40, 3)
    good = tmp_path / "ring.edp"
    edp.edp_save(src.ctx, str(good))
    # a non-empty destination
    with pytest.raises(edp.EdpError) as e:
        edp.edp_load(src.ctx, str(good))
    assert e.value.status == edp.EDP_ERR_STATE
    # another layout
    other = MirroredDqn(64)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_load(other.ring.ctx, str(good))
    assert e.value.status == edp.EDP_ERR_STATE
    # a foreign file and a truncated one leave the context empty
    bogus = tmp_path / "bogus.edp"
    bogus.write_bytes(b"not a checkpoint" * 8)
    cut = tmp_path / "cut.edp"
    cut.write_bytes(good.read_bytes()[:-1000])
    for f in (bogus, cut, tmp_path / "missing.edp"):
        dst = _mm_ring(edp, 64, 24)
        with pytest.raises(edp.EdpError) as e:
            edp.edp_load(dst.ctx, str(f))
        assert e.value.status == edp.EDP_ERR_INVALID
        assert dst.info().total == 0


def test_failed_load_leaves_prioritized_context_empty(edp_lib, orc, tmp_path):
    """A truncated or padded checkpoint is refused before anything reaches
    the context; the context then works as a fresh one (every leaf and sum,
    the deferred and running-maximum priorities)."""
    edp = edp_lib
    Fb = 84 * 16
    frames, action, reward, done = fx.dqn_transitions(71, 700, Fb, done_p=0.05)
    q = orc.priorities_from_td(fx.td_errors(71, 700), 0.6, 1e-6)
    src = MirroredDqn(500, prioritized=True, F=Fb)
    src.ingest(orc, frames[:400], action[:400], reward[:400], done[:400], q=q[:400])
    src.ingest(orc, frames[400:600], action[400:600], reward[400:600], done[400:600],
               q=q[400:600])
    good = tmp_path / "per.edp"
    edp.edp_save(src.ring.ctx, str(good))
    raw = good.read_bytes()
    cut = tmp_path / "cut.edp"
    cut.write_bytes(raw[:-100])  # ends inside the leaves
    pad = tmp_path / "pad.edp"
    pad.write_bytes(raw + bytes(4))
    dst = MirroredDqn(500, prioritized=True, F=Fb)
    for f in (cut, pad):
        with pytest.raises(edp.EdpError) as e:
            edp.edp_load(dst.ring.ctx, str(f))
        assert e.value.status == edp.EDP_ERR_INVALID
        assert dst.ring.info().total == 0
    sl = slice(600, 700)
    dst.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
    edp.edp_sync(dst.ring.ctx)
    check_tree(orc, dst.ring, dst.st)
    # and the intact file still loads into a fresh context
    fresh = MirroredDqn(500, prioritized=True, F=Fb)
    edp.edp_load(fresh.ring.ctx, str(good))
    edp.edp_sync(fresh.ring.ctx)
    assert fresh.ring.info().total == 500
