"""Deliveries into page-locked host memory (the kernel writes the learner
batch over the host link): bit-identical to the same deliveries into device
memory, for the three transforms -- frame stacks with collate and
importance weights, HWC -> CHW bf16 with gathered advantages and returns,
normalised bf16 with tokens from a two-tier ring -- and pageable host
outputs rejected."""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, cuda, dqn_outputs, fx
from test_gpu_mm import C, H, L, W, Logical, _ingest, _mm_ring

pytestmark = pytest.mark.gpu


def _pinned_like(t):
    return torch.empty(t.shape, dtype=t.dtype, pin_memory=True)


def _same(dev, host):
    for x, y in zip(dev, host):
        assert np.array_equal(bits(x).reshape(-1), bits(y).reshape(-1))


def test_frame_stack_per_into_host(edp_lib, orc):
    edp = edp_lib
    frames, action, reward, done = fx.dqn_transitions(21, 1500, done_p=0.05)
    q = orc.priorities_from_td(fx.td_errors(21, 1500), 0.6, 1e-6)
    m = MirroredDqn(1200, prioritized=True)
    for sl in (slice(0, 700), slice(700, 1500)):  # wraps the ring
        m.ingest(orc, frames[sl], action[sl], reward[sl], done[sl], q=q[sl])
    for B in (32, 700):  # one chunk per CTA, and the staged path
        idx = torch.empty(B, dtype=torch.int64, device="cuda")
        qs = torch.empty(B, dtype=torch.int32, device="cuda")
        edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, B, 5, B, idx, qs)
        dev = list(dqn_outputs(B, 4, m.F)) + [torch.empty(B, device="cuda")]
        host = [_pinned_like(t) for t in dev]
        for o in (dev, host):
            edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(*o[:5], q=qs, isw=o[5],
                                                               beta=0.4))
        edp.edp_sync(m.ring.ctx)
        _same(dev, host)


def test_hwc_gathers_into_host(edp_lib):
    edp = edp_lib
    T, E = 16, 32
    n = T * E
    obs, r, v, d = fx.ppo_rollout(6, T, E)
    cfg = edp.make_config(n, (3, 64, 64), edp.EDP_XFORM_HWC_CHW_BF16)
    ring = edp.Ring(cfg, action=False, reward=False, done=False)
    edp.edp_ingest(ring.ctx, torch.from_numpy(obs.reshape(n, -1)).cuda(), n)
    src_a, src_r = cuda(r.reshape(-1)), cuda(v[:T].reshape(-1))
    B = 300
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 3, 1, idx)
    dev = [torch.empty((B, 3, 64, 64), dtype=torch.bfloat16, device="cuda"),
           torch.empty(B, device="cuda"), torch.empty(B, device="cuda")]
    host = [_pinned_like(t) for t in dev]
    for o in (dev, host):
        edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(o[0], gather=[(src_a, o[1]),
                                                                      (src_r, o[2])]))
    edp.edp_sync(ring.ctx)
    _same(dev, host)


def test_two_tier_norm_into_host(edp_lib, orc):
    edp = edp_lib
    ring = _mm_ring(edp, 64, 24)
    lg = Logical(64, 8)
    for n in [30, 50, 24]:
        _ingest(edp, ring, lg, orc, n, 8)
    B = 48
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 2, 6, idx)
    dev = [torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda"),
           torch.empty((B, L), dtype=torch.int32, device="cuda"),
           torch.empty(B, device="cuda")]
    host = [_pinned_like(t) for t in dev]
    for o in (dev, host):
        edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(o[0], tokens=o[1], reward=o[2]))
    edp.edp_sync(ring.ctx)
    _same(dev, host)
    # pageable host memory is not accepted
    with pytest.raises(edp.EdpError) as e:
        edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(torch.empty((B, C, H, W),
                                                                     dtype=torch.bfloat16)))
    assert e.value.status == edp.EDP_ERR_INVALID
