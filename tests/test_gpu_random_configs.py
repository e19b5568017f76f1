"""Randomised configurations against the oracle, to reach the corners of
the launch logic the fixed-size tests do not: frame stacks of K = 1..16 with
and without next_obs, frame sizes of one and several shared-memory pieces,
dense and sparse episode ends, rings filled in random chunk sizes past a wrap
(insertions take the one-launch path up to 16,384 rows, the kernel chain
above), batches on both sides of the staged delivery's threshold; and
normalised deliveries of 1 to 4 channels, with and without tokens, on one
and two tiers.  Every output bit-exact against the oracle."""
import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, to_np

pytestmark = pytest.mark.gpu


def _stack_case(edp, orc, seed):
    rng = np.random.default_rng(1000 + seed)
    K = int(rng.integers(1, 17))
    nxt = bool(rng.integers(0, 2))
    w = int(rng.choice([20, 84, 112]))  # 84 x w bytes per frame: 1 or 2 pieces
    F = 84 * w
    cap = int(rng.integers(40, 2500))
    done_p = float(rng.choice([0.0, 0.02, 0.3]))
    prioritized = bool(rng.integers(0, 2))
    cfg = edp.make_config(cap, (1, 84, w), edp.EDP_XFORM_STACK_F32, frame_stack=K,
                          next_obs=nxt, prioritized=prioritized)
    ring = edp.Ring(cfg)
    total_n = int(cap * rng.uniform(0.5, 2.5)) + 2
    frames = rng.integers(0, 256, size=(total_n, F), dtype=np.uint8)
    action = rng.integers(0, 6, size=total_n).astype(np.int32)
    reward = rng.standard_normal(total_n).astype(np.float32)
    done = (rng.random(total_n) < done_p).astype(np.uint8)
    q = rng.integers(1, 1 << 22, size=total_n).astype(np.uint32)
    o_frames = np.zeros((cap, F), np.uint8)
    o_act = np.zeros(cap, np.int32)
    o_rew = np.zeros(cap, np.float32)
    o_done = np.zeros(cap, np.uint8)
    st = orc.PerState(cap, nxt) if prioritized else None
    t = 0
    while t < total_n:
        n = int(min(total_n - t, rng.integers(1, cap + 1)))
        sl = slice(t, t + n)
        edp.edp_ingest(ring.ctx, cuda(frames[sl]), n, action=cuda(action[sl]),
                       reward=cuda(reward[sl]), done=cuda(done[sl]),
                       q=cuda(q[sl].view(np.int32)) if prioritized else None)
        for a, src in [(o_frames, frames), (o_act, action), (o_rew, reward), (o_done, done)]:
            orc.ring_write(a, cap, t, np.ascontiguousarray(src[sl]))
        if prioritized:
            orc.ingest_leaves(st, t, q[sl])
        t += n
    size = min(t, cap)
    n_valid = size - (1 if nxt else 0)
    if n_valid <= 0:
        ring.close()
        return
    for B in (int(rng.integers(1, 40)), int(rng.integers(150, 700))):
        idx = torch.empty(B, dtype=torch.int64, device="cuda")
        if prioritized:
            qs = torch.empty(B, dtype=torch.int32, device="cuda")
            edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, B, seed, B, idx, qs)
            ref_idx, ref_q = orc.sample_prioritized_bisect(st.leaves, B, seed, B)
        else:
            edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, seed, B, idx)
            ref_idx = orc.sample_uniform(cap, t, n_valid, B, seed, B)
        obs = torch.full((B, K, F), float("nan"), device="cuda")
        nx = torch.full((B, K, F), float("nan"), device="cuda") if nxt else None
        act = torch.full((B,), -3, dtype=torch.int32, device="cuda")
        rew = torch.full((B,), float("nan"), device="cuda")
        dn = torch.full((B,), 7, dtype=torch.uint8, device="cuda")
        edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(obs, nx, act, rew, dn))
        edp.edp_sync(ring.ctx)
        assert np.array_equal(to_np(idx), ref_idx), (seed, B)
        if prioritized:
            assert np.array_equal(to_np(qs).view(np.uint32), ref_q), (seed, B)
        r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
            o_frames, o_done, o_act, o_rew, cap, t, K, ref_idx, with_next=nxt)
        assert np.array_equal(bits(obs).reshape(r_obs.shape), r_obs.view(np.uint32)), (seed, B)
        if nxt:
            assert np.array_equal(bits(nx).reshape(r_nxt.shape), r_nxt.view(np.uint32)), (seed, B)
        assert np.array_equal(to_np(act), r_act) and np.array_equal(to_np(dn), r_dn)
        assert np.array_equal(bits(rew), r_rew.view(np.uint32))
    ring.close()


@pytest.mark.parametrize("seed", range(40))
def test_random_frame_stack_configs(edp_lib, orc, seed):
    _stack_case(edp_lib, orc, seed)


@pytest.mark.parametrize("seed", range(30))
def test_random_normalised_configs(edp_lib, orc, seed):
    edp = edp_lib
    rng = np.random.default_rng(2000 + seed)
    C = int(rng.integers(1, 5))
    H, W = int(rng.choice([4, 16, 32])), int(rng.choice([4, 16, 40]))
    if (H * W) % 16:
        W = 16
    L = int(rng.choice([0, 4, 64]))
    cap = int(rng.integers(8, 300))
    cap_h = cap if rng.random() < 0.5 else int(rng.integers(1, cap + 1))
    mean = tuple(float(x) for x in rng.uniform(0.2, 0.8, 4))
    std = tuple(float(x) for x in rng.uniform(0.1, 0.4, 4))
    cfg = edp.make_config(cap, (C, H, W), edp.EDP_XFORM_CHW_NORM_BF16, hbm_capacity=cap_h,
                          tokens=L, norm_mean=mean, norm_std=std)
    ring = edp.Ring(cfg, action=False, done=False)
    F = C * H * W
    total_n = int(cap * rng.uniform(0.5, 3.0)) + 1
    img = rng.integers(0, 256, size=(total_n, F), dtype=np.uint8)
    tok = rng.integers(0, 32000, size=(total_n, max(L, 1)), dtype=np.int32)[:, :L]
    rew = rng.standard_normal(total_n).astype(np.float32)
    o_img = np.zeros((cap, F), np.uint8)
    o_tok = np.zeros((cap, L), np.int32)
    o_rew = np.zeros(cap, np.float32)
    t = 0
    while t < total_n:
        n = int(min(total_n - t, rng.integers(1, cap + 1)))
        sl = slice(t, t + n)
        edp.edp_ingest(ring.ctx, cuda(img[sl]), n,
                       tokens=cuda(np.ascontiguousarray(tok[sl])) if L else None,
                       reward=cuda(rew[sl]))
        orc.ring_write(o_img, cap, t, np.ascontiguousarray(img[sl]))
        if L:
            orc.ring_write(o_tok, cap, t, np.ascontiguousarray(tok[sl]))
        orc.ring_write(o_rew, cap, t, np.ascontiguousarray(rew[sl]))
        t += n
    size = min(t, cap)
    for B in (int(rng.integers(1, 20)), int(rng.integers(100, 800))):
        idx = torch.empty(B, dtype=torch.int64, device="cuda")
        out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
        otok = torch.full((B, L), -1, dtype=torch.int32, device="cuda") if L else None
        orew = torch.empty(B, device="cuda")
        edp.edp_sample_deliver(ring.ctx, B, seed, B, idx,
                               edp.make_batch(out, tokens=otok, reward=orew))
        edp.edp_sync(ring.ctx)
        ref_idx = orc.sample_uniform(cap, t, size, B, seed, B)
        assert np.array_equal(to_np(idx), ref_idx), (seed, B)
        r_img, r_tok, r_rew = orc.deliver_mm(o_img, o_tok if L else None, o_rew, C, H * W,
                                             ref_idx, mean[:C], std[:C])
        assert np.array_equal(bits(out).reshape(B, -1), r_img), (seed, B)
        if L:
            assert np.array_equal(to_np(otok), r_tok), (seed, B)
        assert np.array_equal(bits(orew), r_rew.view(np.uint32)), (seed, B)
    ring.close()
