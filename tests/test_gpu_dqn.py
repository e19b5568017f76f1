"""GPU parity of the off-policy path through the C ABI: ring scatter,
Philox uniform sampling, and the fused frame-stack delivery, against the
oracle (indices and bytes bit-exact, fp32 bit-exact)."""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, dqn_outputs, fx, to_np

pytestmark = pytest.mark.gpu


def _deliver_and_check(edp, orc, m, B, seed, rnd, with_next=True):
    idx = torch.full((B,), -5, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, seed, rnd, idx)
    obs, nxt, act, rew, dn = dqn_outputs(B, m.K, m.F, with_next)
    edp.edp_deliver(m.ring.ctx, idx, B,
                    edp.make_batch(obs, nxt, act, rew, dn))
    edp.edp_sync(m.ring.ctx)
    size = min(m.total, m.cap)
    n_valid = size - (1 if with_next else 0)
    ref_idx = orc.sample_uniform(m.cap, m.total, n_valid, B, seed, rnd)
    assert np.array_equal(to_np(idx), ref_idx)
    r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
        m.frames, m.done, m.action, m.reward, m.cap, m.total, m.K, ref_idx,
        with_next=with_next)
    assert np.array_equal(bits(obs).reshape(r_obs.shape), r_obs.view(np.uint32))
    if with_next:
        assert np.array_equal(bits(nxt).reshape(r_nxt.shape), r_nxt.view(np.uint32))
    assert np.array_equal(to_np(act), r_act)
    assert np.array_equal(bits(rew), r_rew.view(np.uint32))
    assert np.array_equal(to_np(dn), r_dn)


def test_dqn_uniform_ragged_wrap(edp_lib, orc):
    edp = edp_lib
    cap = 1000
    frames, action, reward, done = fx.dqn_transitions(0, 2500, done_p=0.05)
    m = MirroredDqn(cap)
    t = 0
    for n in [1, 998, 3, 600, 898]:
        sl = slice(t, t + n)
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl])
        t += n
        if m.total == 1:  # no transition has a successor yet
            idx = torch.empty(4, dtype=torch.int64, device="cuda")
            with pytest.raises(edp.EdpError) as e:
                edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, 4, 0, 0, idx)
            assert e.value.status == edp.EDP_ERR_EMPTY
            continue
        _deliver_and_check(edp, orc, m, 37, seed=5, rnd=m.total)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_dqn_tiny_config(edp_lib, orc, seed):
    """Capacity 10,000 uniform-byte 84x84 frames, filled past capacity so the
    wrap is exercised; batches of 32 for several rounds."""
    cap = 10_000
    frames, action, reward, done = fx.dqn_transitions(seed, 12_345)
    m = MirroredDqn(cap)
    for lo in range(0, 12_345, 4096):
        hi = min(12_345, lo + 4096)
        m.ingest(orc, frames[lo:hi], action[lo:hi], reward[lo:hi], done[lo:hi])
    for rnd in range(4):
        _deliver_and_check(edp_lib, orc, m, 32, seed=seed, rnd=rnd)


@pytest.mark.parametrize("K,with_next", [(1, True), (2, False), (4, False), (7, True)])
def test_dqn_stack_variants(edp_lib, orc, K, with_next):
    cap = 300
    frames, action, reward, done = fx.dqn_transitions(7, 450, done_p=0.2)
    m = MirroredDqn(cap, K=K, next_obs=with_next)
    m.ingest(orc, frames[:200], action[:200], reward[:200], done[:200])
    _deliver_and_check(edp_lib, orc, m, 513, seed=3, rnd=0, with_next=with_next)
    m.ingest(orc, frames[200:], action[200:], reward[200:], done[200:])
    _deliver_and_check(edp_lib, orc, m, 64, seed=3, rnd=1, with_next=with_next)


def test_dqn_all_byte_values(edp_lib, orc):
    """Every byte value through the fp32 transform, bit-exact."""
    cap, n = 64, 64
    F = 84 * 84
    frames = (np.arange(n * F) % 256).astype(np.uint8).reshape(n, F)
    action = np.zeros(n, np.int32)
    reward = np.zeros(n, np.float32)
    done = np.zeros(n, np.uint8)
    m = MirroredDqn(cap)
    m.ingest(orc, frames, action, reward, done)
    _deliver_and_check(edp_lib, orc, m, 200, seed=9, rnd=9)
    lut = np.array([orc.unit_f32(b) for b in range(256)], np.float32)
    assert np.array_equal(lut, np.arange(256, dtype=np.float32) / np.float32(255))


def test_dqn_host_pinned_ingest_source(edp_lib, orc):
    """An ingest source in page-locked host memory is read over the host
    link with the same result."""
    edp = edp_lib
    cap = 128
    frames, action, reward, done = fx.dqn_transitions(3, 100)
    m = MirroredDqn(cap)
    pf = torch.from_numpy(frames).pin_memory()
    edp.edp_ingest(m.ring.ctx, pf, 100, action=torch.from_numpy(action).pin_memory(),
                   reward=torch.from_numpy(reward).pin_memory(),
                   done=torch.from_numpy(done).pin_memory())
    for arr, src in [(m.frames, frames), (m.action, action), (m.reward, reward),
                     (m.done, done)]:
        orc.ring_write(arr, cap, 0, np.ascontiguousarray(src))
    m.total = 100
    _deliver_and_check(edp, orc, m, 50, seed=1, rnd=2)


@pytest.mark.parametrize("fw", [112, 560])
def test_staged_stack_multi_piece_frames_and_bad_indices(edp_lib, orc, fw):
    """Frames larger than one shared-memory stage (84 x 112 = 9,408 B in two
    pieces, 84 x 560 = 47,040 B in seven) through the staged delivery (a
    batch of 300 stacks fills the GPU), with episode ends and a wrapped ring;
    slots outside the sampleable range (-1, capacity, the newest slot, whose
    successor does not exist) give zero rows and a device flag, and every
    other row equals the oracle's."""
    edp = edp_lib
    cap, n, B = 700, 900, 300
    F = 84 * fw
    frames, action, reward, done = fx.dqn_transitions(11, n, frame_bytes=F, done_p=0.1)
    m = MirroredDqn(cap, F=F)
    m.ingest(orc, frames[:500], action[:500], reward[:500], done[:500])
    m.ingest(orc, frames[500:], action[500:], reward[500:], done[500:])
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 4, 0, idx)
    newest = (m.total - 1) % cap
    bad = {7: -1, 100: cap, 211: newest}
    for k, v in bad.items():
        idx[k] = v
    obs, nxt, act, rew, dn = dqn_outputs(B, m.K, m.F)
    edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(obs, nxt, act, rew, dn))
    st, msg = edp.edp_sync_status(m.ring.ctx)
    assert st == edp.EDP_ERR_INVALID, msg
    got = to_np(idx)
    good = np.array([k for k in range(B) if k not in bad])
    r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
        m.frames, m.done, m.action, m.reward, m.cap, m.total, m.K, got[good])
    o, x = bits(obs).reshape(B, -1), bits(nxt).reshape(B, -1)
    assert np.array_equal(o[good], r_obs.reshape(len(good), -1).view(np.uint32))
    assert np.array_equal(x[good], r_nxt.reshape(len(good), -1).view(np.uint32))
    assert np.array_equal(to_np(act)[good], r_act)
    assert np.array_equal(bits(rew)[good], r_rew.view(np.uint32))
    assert np.array_equal(to_np(dn)[good], r_dn)
    for k in bad:
        assert not o[k].any() and not x[k].any(), k
        assert to_np(act)[k] == 0 and bits(rew)[k] == 0 and to_np(dn)[k] == 0, k
