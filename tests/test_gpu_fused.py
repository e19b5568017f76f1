"""The fused uniform sample -> deliver call (edp_sample_deliver) through the
C ABI: the same indices as edp_sample(UNIFORM) with the same seed and round
(and as the oracle's sampler), and outputs bit-identical to edp_deliver of
those indices, for the three transforms -- frame stacks (one chunk per CTA
and the staged path), HWC -> CHW bf16, and normalised bf16 over a
two-tier ring; plus its argument errors."""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, dqn_outputs, fx, to_np
from test_gpu_mm import Logical, _ingest, _mm_ring, C, H, W, L

pytestmark = pytest.mark.gpu


def _same(a, b):
    for x, y in zip(a, b):
        if x is None:
            continue
        assert np.array_equal(bits(x) if x.is_floating_point() else to_np(x),
                              bits(y) if y.is_floating_point() else to_np(y))


@pytest.mark.parametrize("B", [37, 600])
def test_fused_frame_stack(edp_lib, orc, B):
    edp = edp_lib
    frames, action, reward, done = fx.dqn_transitions(60, 2600, done_p=0.05)
    m = MirroredDqn(1000)
    t = 0
    for n in [700, 900, 1000]:  # wraps the ring
        sl = slice(t, t + n)
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl])
        t += n
    idx_a = torch.empty(B, dtype=torch.int64, device="cuda")
    idx_b = torch.full((B,), -3, dtype=torch.int64, device="cuda")
    a = dqn_outputs(B, 4, m.F)
    b = dqn_outputs(B, 4, m.F)
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 9, 4, idx_a)
    edp.edp_deliver(m.ring.ctx, idx_a, B, edp.make_batch(*a))
    edp.edp_sample_deliver(m.ring.ctx, B, 9, 4, idx_b, edp.make_batch(*b))
    edp.edp_sync(m.ring.ctx)
    ref = orc.sample_uniform(m.cap, m.total, min(m.total, m.cap) - 1, B, 9, 4)
    assert np.array_equal(to_np(idx_b), ref)
    assert np.array_equal(to_np(idx_a), ref)
    _same(a, b)


def test_fused_hwc(edp_lib):
    edp = edp_lib
    T, E, Hh, Ww, Cc = 16, 32, 64, 64, 3
    n = T * E
    obs, _, _, _ = fx.ppo_rollout(5, T, E)
    cfg = edp.make_config(n, (Cc, Hh, Ww), edp.EDP_XFORM_HWC_CHW_BF16)
    ring = edp.Ring(cfg, action=False, reward=False, done=False)
    edp.edp_ingest(ring.ctx, torch.from_numpy(obs.reshape(n, -1)).cuda(), n)
    B = 300
    idx_a = torch.empty(B, dtype=torch.int64, device="cuda")
    idx_b = torch.empty(B, dtype=torch.int64, device="cuda")
    oa = torch.empty((B, Cc, Hh, Ww), dtype=torch.bfloat16, device="cuda")
    ob = torch.empty_like(oa)
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 3, 1, idx_a)
    edp.edp_deliver(ring.ctx, idx_a, B, edp.make_batch(oa))
    edp.edp_sample_deliver(ring.ctx, B, 3, 1, idx_b, edp.make_batch(ob))
    edp.edp_sync(ring.ctx)
    assert np.array_equal(to_np(idx_a), to_np(idx_b))
    assert np.array_equal(bits(oa), bits(ob))


def test_fused_two_tier(edp_lib, orc):
    edp = edp_lib
    ring = _mm_ring(edp, 64, 24)
    lg = Logical(64, 8)
    for n in [30, 50, 24]:
        _ingest(edp, ring, lg, orc, n, 8)
    B = 48
    outs = []
    for _ in range(2):
        outs.append((torch.empty(B, dtype=torch.int64, device="cuda"),
                     torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda"),
                     torch.full((B, L), -1, dtype=torch.int32, device="cuda"),
                     torch.full((B,), float("nan"), device="cuda")))
    (ia, oa, ta, ra), (ib, ob, tb, rb) = outs
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 2, 6, ia)
    edp.edp_deliver(ring.ctx, ia, B, edp.make_batch(oa, tokens=ta, reward=ra))
    edp.edp_sample_deliver(ring.ctx, B, 2, 6, ib, edp.make_batch(ob, tokens=tb, reward=rb))
    edp.edp_sync(ring.ctx)
    ref = orc.sample_uniform(lg.cap, lg.total, min(lg.total, lg.cap), B, 2, 6)
    assert np.array_equal(to_np(ib), ref)
    _same((ia, oa, ta, ra), (ib, ob, tb, rb))


def test_fused_argument_errors(edp_lib, orc):
    edp = edp_lib
    m = MirroredDqn(100)
    B = 4
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    out = dqn_outputs(B, 4, m.F)
    with pytest.raises(edp.EdpError) as e:  # nothing stored yet
        edp.edp_sample_deliver(m.ring.ctx, B, 1, 0, idx, edp.make_batch(*out))
    assert e.value.status == edp.EDP_ERR_EMPTY
    frames, action, reward, done = fx.dqn_transitions(61, 50)
    m.ingest(orc, frames, action, reward, done)
    q = torch.zeros(B, dtype=torch.int32, device="cuda")
    isw = torch.zeros(B, device="cuda")
    with pytest.raises(edp.EdpError) as e:  # uniform draws carry no priorities
        edp.edp_sample_deliver(m.ring.ctx, B, 1, 0, idx,
                               edp.make_batch(*out, q=q, isw=isw, beta=0.4))
    assert e.value.status == edp.EDP_ERR_INVALID
