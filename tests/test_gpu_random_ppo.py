"""Randomised on-policy cases against the oracle: the shuffle at sizes up
to twice the 32,768-element rollout (so that buckets hold more than their
usual four keys) with random seeds, iterations and ring offsets, bit-exact;
GAE over random shapes, episode-end rates and discounts, within 1e-5 of
the fp64 oracle (advantages, returns, normalised advantages)."""
import numpy as np
import pytest
import torch

from gpu_util import cuda, fx, to_np

pytestmark = pytest.mark.gpu


def _ring(edp, cap, H=4, W=4, C=1):
    cfg = edp.make_config(cap, (C, H, W), edp.EDP_XFORM_HWC_CHW_BF16)
    return edp.Ring(cfg, action=False, reward=False, done=False)


@pytest.mark.parametrize("seed", range(12))
def test_random_shuffles(edp_lib, orc, seed):
    edp = edp_lib
    rng = np.random.default_rng(8000 + seed)
    n = int(rng.choice([int(rng.integers(1, 64)), int(rng.integers(64, 5000)),
                        int(rng.integers(30000, 70000))]))
    extra = int(rng.integers(0, n + 1))  # ring offset: insertions before the rollout
    cap = n
    ring = _ring(edp, cap)
    if extra:
        edp.edp_ingest(ring.ctx, cuda(np.zeros((extra, 16), np.uint8)), extra)
    edp.edp_ingest(ring.ctx, cuda(np.zeros((n, 16), np.uint8)), n)
    s, it = int(rng.integers(0, 1 << 40)), int(rng.integers(0, 1 << 20))
    idx = torch.full((n,), -1, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, n, s, it, idx)
    edp.edp_sync(ring.ctx)
    perm = orc.permutation(n, s, it)
    oldest = (extra + n - n) % cap  # total = extra + n, size = n
    assert np.array_equal(to_np(idx), (oldest + perm) % cap), (n, extra)
    ring.close()


@pytest.mark.parametrize("seed", range(12))
def test_random_gae(edp_lib, orc, seed):
    edp = edp_lib
    rng = np.random.default_rng(9000 + seed)
    T, E = int(rng.integers(1, 400)), int(rng.integers(1, 600))
    done_p = float(rng.choice([0.0, 0.003, 0.05, 0.5, 1.0]))
    gamma, lam = float(rng.uniform(0.9, 0.999)), float(rng.uniform(0.8, 1.0))
    _, r, v, d = fx.ppo_rollout(9000 + seed, T, E, done_p=done_p, with_obs=False)
    ring = _ring(edp, 64)
    adv = torch.full((T, E), float("nan"), device="cuda")
    ret = torch.full((T, E), float("nan"), device="cuda")
    nrm = torch.full((T, E), float("nan"), device="cuda")
    edp.edp_gae(ring.ctx, cuda(r), cuda(v), cuda(d), T, E, gamma, lam, adv, ret, nrm)
    edp.edp_sync(ring.ctx)
    ra, rr = orc.gae(r, v, d, gamma, lam)
    rn, _, _ = orc.normalize(ra.ravel())
    assert np.abs(to_np(adv) - ra).max() <= 1e-5, (T, E, done_p)
    assert np.abs(to_np(ret) - rr).max() <= 1e-5
    assert np.abs(to_np(nrm).ravel() - rn).max() <= 1e-5
    ring.close()
