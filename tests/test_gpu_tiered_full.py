"""Two-tier parity at the size the benchmark times: 1,600,000 transitions
of 3x224x224 images + 512 tokens, the newest 800,000 in HBM (122 GB) and
the oldest 800,000 in page-locked host memory (122 GB), 4,096 transitions
ingested per step from page-locked staging (the steady-state path where
each new transition takes the HBM slot of the one it demotes), uniform batch
1,024 read from both tiers.  Checked every step: all indices against the
oracle's sampler, a strided subset of delivered samples (image, tokens,
reward) against the content function of their logical ids, and a sample of
retained ids in the tier and slot the placement map gives."""
import gc

import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, fx, to_np
from test_gpu_mm import C, F, H, L, MEAN, STD, W, _mm_ring

pytestmark = pytest.mark.gpu

CAP, CAP_H, SEED, B, STEP = 1_600_000, 800_000, 1240, 1024, 4096


def test_two_tier_full_size(edp_lib, orc):
    edp = edp_lib
    ring = _mm_ring(edp, CAP, CAP_H)
    steps = 3
    _, rew_all = fx.mm_metadata(SEED, CAP + steps * STEP, tokens=0)
    try:
        chunk = 8192
        obs = torch.empty((chunk, F), dtype=torch.uint8, device="cuda")
        tok = torch.empty((chunk, L), dtype=torch.int32, device="cuda")
        for lo in range(0, CAP, chunk):
            n = min(chunk, CAP - lo)
            fx.content_fill_torch(SEED, lo, obs[:n])
            fx.token_fill_torch(SEED, lo, tok[:n])
            edp.edp_ingest(ring.ctx, obs[:n], n, tokens=tok[:n],
                           reward=cuda(rew_all[lo:lo + n]))
        edp.edp_sync(ring.ctx)
        st_obs = torch.empty((STEP, F), dtype=torch.uint8, pin_memory=True)
        st_tok = torch.empty((STEP, L), dtype=torch.int32, pin_memory=True)
        total = CAP
        rng = np.random.default_rng(SEED)
        for step in range(steps):
            # the step's new transitions, staged in page-locked host memory
            fx.content_fill_torch(SEED, total, obs[:STEP])
            fx.token_fill_torch(SEED, total, tok[:STEP])
            st_obs.copy_(obs[:STEP])
            st_tok.copy_(tok[:STEP])
            edp.edp_ingest(ring.ctx, st_obs, STEP, tokens=st_tok,
                           reward=cuda(rew_all[total:total + STEP]))
            total += STEP
            idx = torch.empty(B, dtype=torch.int64, device="cuda")
            edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 31, step, idx)
            out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
            tk = torch.full((B, L), -1, dtype=torch.int32, device="cuda")
            rw = torch.full((B,), float("nan"), device="cuda")
            edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(out, tokens=tk, reward=rw))
            edp.edp_sync(ring.ctx)
            assert ring.info().total == total
            ref_idx = orc.sample_uniform(CAP, total, CAP, B, 31, step)
            assert np.array_equal(to_np(idx), ref_idx)
            # logical id of a slot: the full ring holds ids total-CAP .. total-1
            oldest = total % CAP
            ids = total - CAP + (ref_idx - oldest) % CAP
            assert ((ids % CAP) == ref_idx).all()
            sel = np.arange(step, B, 29)
            r_obs, r_tok, r_rew = orc.deliver_mm(
                fx.content_bytes(SEED, ids[sel], F), fx.token_content(SEED, ids[sel], L),
                rew_all[ids[sel]], C, H * W, np.arange(len(sel)), MEAN, STD)
            assert np.array_equal(bits(out).reshape(B, -1)[sel], r_obs)
            assert np.array_equal(to_np(tk)[sel], r_tok)
            assert np.array_equal(bits(rw)[sel], r_rew.view(np.uint32))
            # placement of retained ids, including both ends of each tier
            probe = np.concatenate([
                [total - CAP, total - CAP_H - 1, total - CAP_H, total - 1],
                rng.integers(total - CAP, total, size=12)])
            for Lid in probe:
                tier, slot = orc.tier_of(CAP, CAP_H, total, int(Lid))
                row = (ring.host_obs[slot].numpy() if tier == 1
                       else ring.obs[slot].cpu().numpy())
                assert tier == (0 if Lid >= total - CAP_H else 1), Lid
                assert np.array_equal(row, fx.content_bytes(SEED, [int(Lid)], F)[0]), Lid
    finally:
        ring.close()
        del ring
        gc.collect()
        torch.cuda.empty_cache()
        if hasattr(torch._C, "_host_emptyCache"):
            torch._C._host_emptyCache()  # the 122 GB of page-locked host tier
