"""The per-context traffic counters (edp_get_counters) against the byte
counts of the calls made: insertions from device and from page-locked host
sources, prioritized sampling, frame-stack deliveries into device and into
host outputs, TD-error updates; and a two-tier ring, whose delivery counts
its host-tier rows on the device -- the rows the oracle's tier map puts in
the host tier for the sampled slots."""
import numpy as np
import pytest
import torch

from gpu_util import cuda, to_np

pytestmark = pytest.mark.gpu


def test_counters_stack_ring(edp_lib, orc):
    from paper_2609_24456_gb300 import fixtures as fx
    edp = edp_lib
    cap, K, F = 1000, 4, 84 * 84
    cfg = edp.make_config(cap, (1, 84, 84), edp.EDP_XFORM_STACK_F32, frame_stack=K,
                          next_obs=True, prioritized=True)
    ring = edp.Ring(cfg)  # action, reward, done and the leaves in HBM
    ctx = ring.ctx
    assert all(v == 0 for v in edp.edp_get_counters(ctx).values())
    frames, action, reward, done = fx.dqn_transitions(5, 900)
    q = orc.priorities_from_td(fx.td_errors(5, 900), 0.6, 1e-6)
    meta_ring = 4 + 4 + 1 + 4
    # 600 from device memory, 300 from page-locked host memory
    edp.edp_ingest(ctx, cuda(frames[:600]), 600, action=cuda(action[:600]),
                   reward=cuda(reward[:600]), done=cuda(done[:600]), q=cuda(q[:600].view(np.int32)))
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    edp.edp_ingest(ctx, pin(frames[600:]), 300, action=pin(action[600:]),
                   reward=pin(reward[600:]), done=pin(done[600:]))
    want = dict(calls=2, ingested=900, sampled=0, delivered=0,
                hbm_read=600 * (F + 4 + 4 + 1 + 4), hbm_write=900 * (F + meta_ring),
                link_read=300 * (F + 4 + 4 + 1), link_write=0)
    assert edp.edp_get_counters(ctx) == want
    B = 64
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    qs = torch.empty(B, dtype=torch.int32, device="cuda")
    edp.edp_sample(ctx, edp.EDP_SAMPLE_PRIORITIZED, B, 2, 0, idx, qs)
    want["calls"] += 1
    want["sampled"] += B
    want["hbm_write"] += 12 * B
    dev_out = [torch.empty((B, K, F), device="cuda"), torch.empty((B, K, F), device="cuda"),
               torch.empty(B, dtype=torch.int32, device="cuda"), torch.empty(B, device="cuda"),
               torch.empty(B, dtype=torch.uint8, device="cuda")]
    isw = torch.empty(B, device="cuda")
    edp.edp_deliver(ctx, idx, B, edp.make_batch(*dev_out, q=qs, isw=isw, beta=0.4))
    per_read = (K + 1) * F + 8 + 4 + 4 + 1 + 4
    per_write = 2 * K * F * 4 + 4 + 4 + 1 + 4
    want["calls"] += 1
    want["delivered"] += B
    want["hbm_read"] += B * per_read
    want["hbm_write"] += B * per_write
    host_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in dev_out]
    edp.edp_deliver(ctx, idx, B, edp.make_batch(*host_out))
    want["calls"] += 1
    want["delivered"] += B
    want["hbm_read"] += B * ((K + 1) * F + 8 + 4 + 4 + 1)
    want["link_write"] += B * (2 * K * F * 4 + 4 + 4 + 1)
    edp.edp_update_priorities_td(ctx, idx, cuda(fx.td_errors(5, B, 1)), B, 0.6, 1e-6)
    want["calls"] += 1
    want["hbm_read"] += 12 * B
    want["hbm_write"] += 4 * B
    edp.edp_sync(ctx)
    assert edp.edp_get_counters(ctx) == want
    edp.edp_reset_counters(ctx)
    assert all(v == 0 for v in edp.edp_get_counters(ctx).values())


def test_counters_two_tier_host_rows(edp_lib, orc):
    edp = edp_lib
    cap, cap_h, C, H, W, L = 64, 24, 3, 16, 16, 8
    F, R = C * H * W, C * H * W + 4 * L
    cfg = edp.make_config(cap, (C, H, W), edp.EDP_XFORM_CHW_NORM_BF16, hbm_capacity=cap_h,
                          tokens=L, norm_mean=(0.5,) * 4, norm_std=(0.25,) * 4)
    ring = edp.Ring(cfg, action=False, done=False)
    ctx = ring.ctx
    rng = np.random.default_rng(9)
    n = 100
    img = rng.integers(0, 256, size=(n, F), dtype=np.uint8)
    tok = rng.integers(0, 1000, size=(n, L), dtype=np.int32)
    rew = rng.standard_normal(n).astype(np.float32)
    for lo, hi in [(0, 40), (40, 70), (70, 100)]:  # demotions and evictions
        edp.edp_ingest(ctx, cuda(img[lo:hi]), hi - lo, tokens=cuda(tok[lo:hi]),
                       reward=cuda(rew[lo:hi]))
    edp.edp_reset_counters(ctx)
    B = 50
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
    otok = torch.empty((B, L), dtype=torch.int32, device="cuda")
    orew = torch.empty(B, device="cuda")
    edp.edp_sample(ctx, edp.EDP_SAMPLE_UNIFORM, B, 4, 0, idx)
    edp.edp_deliver(ctx, idx, B, edp.make_batch(out, tokens=otok, reward=orew))
    edp.edp_sync(ctx)
    got = edp.edp_get_counters(ctx)
    total, size = n, cap
    oldest = (total - size) % cap
    host_rows = 0
    for s in to_np(idx):
        L_id = total - size + (int(s) - oldest) % cap
        tier, _ = orc.tier_of(cap, cap_h, total, L_id)
        host_rows += tier == 1
    assert 0 < host_rows < B
    read_all = B * (R + 8 + 4)
    assert got["link_read"] == host_rows * R
    assert got["hbm_read"] == read_all - host_rows * R
    assert got["hbm_write"] == 8 * B + B * (2 * F + 4 * L + 4)
    assert got["delivered"] == B and got["sampled"] == B and got["calls"] == 2
