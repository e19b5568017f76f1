"""GPU parity of the on-policy path through the C ABI: GAE with global
advantage normalisation (within 1e-5 of the fp64 oracle), the Philox
shuffle (bit-exact), and HWC uint8 -> CHW bf16 mini-batch delivery with
gathered advantages and returns (bit-exact)."""
import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, fx, to_np

pytestmark = pytest.mark.gpu

G, LAM = 0.99, 0.95


def _ppo_ring(edp, cap, H=64, W=64, C=3):
    cfg = edp.make_config(cap, (C, H, W), edp.EDP_XFORM_HWC_CHW_BF16)
    return edp.Ring(cfg, action=False, reward=False, done=False)


def _gae(edp, ring, r, v, d, want=(True, True, True)):
    T, E = r.shape
    adv = torch.full((T, E), float("nan"), device="cuda") if want[0] else None
    ret = torch.full((T, E), float("nan"), device="cuda") if want[1] else None
    nrm = torch.full((T, E), float("nan"), device="cuda") if want[2] else None
    edp.edp_gae(ring.ctx, cuda(r), cuda(v), cuda(d), T, E, G, LAM, adv, ret, nrm)
    edp.edp_sync(ring.ctx)
    return adv, ret, nrm


@pytest.mark.parametrize("T,E,done_p", [(128, 256, 0.005), (37, 5, 0.05),
                                        (200, 3, 0.01), (1, 2, 0.5),
                                        (2, 1, 0.0), (300, 130, 0.02),
                                        (129, 8, 1.0),
                                        (5, 512, 0.02), (4, 513, 0.02), (3, 700, 0.01),
                                        (1, 1, 0.0), (1, 1, 1.0)])
def test_gae_matches_oracle(edp_lib, orc, T, E, done_p):
    edp = edp_lib
    _, r, v, d = fx.ppo_rollout(T * 1000 + E, T, E, done_p=done_p, with_obs=False)
    ring = _ppo_ring(edp, 64)
    adv, ret, nrm = _gae(edp, ring, r, v, d)
    ra, rr = orc.gae(r, v, d, G, LAM)
    rn, _, _ = orc.normalize(ra.ravel())
    assert np.abs(to_np(adv) - ra).max() <= 1e-5
    assert np.abs(to_np(ret) - rr).max() <= 1e-5
    assert np.abs(to_np(nrm).ravel() - rn).max() <= 1e-5


def test_gae_single_value_and_bad_shapes(edp_lib, orc):
    # one step of one environment: A = delta, and it normalises to 0
    edp = edp_lib
    ring = _ppo_ring(edp, 64)
    r = np.array([[0.75]], np.float32)
    v = np.array([[0.5], [2.0]], np.float32)
    d = np.zeros((1, 1), np.uint8)
    adv, ret, nrm = _gae(edp, ring, r, v, d)
    delta = 0.75 + G * 2.0 - 0.5
    assert abs(float(adv[0, 0]) - delta) <= 1e-6
    assert abs(float(ret[0, 0]) - (delta + 0.5)) <= 1e-6
    assert float(nrm[0, 0]) == 0.0
    z = torch.zeros(4, device="cuda")
    for T, E in [(0, 4), (4, 0), (1 << 16, 1 << 15)]:
        with pytest.raises(edp.EdpError) as e:
            edp.edp_gae(ring.ctx, z, z, z, T, E, G, LAM, z, None, None)
        assert e.value.status == edp.EDP_ERR_INVALID


def test_gae_optional_outputs(edp_lib, orc):
    edp = edp_lib
    _, r, v, d = fx.ppo_rollout(3, 64, 32, with_obs=False)
    ring = _ppo_ring(edp, 64)
    ra, rr = orc.gae(r, v, d, G, LAM)
    rn, _, _ = orc.normalize(ra.ravel())
    _, ret, nrm = _gae(edp, ring, r, v, d, want=(False, True, True))
    assert np.abs(to_np(nrm).ravel() - rn).max() <= 1e-5
    assert np.abs(to_np(ret) - rr).max() <= 1e-5
    adv, _, _ = _gae(edp, ring, r, v, d, want=(True, False, False))
    assert np.abs(to_np(adv) - ra).max() <= 1e-5


@pytest.mark.parametrize("n", [1, 5, 1000, 32768])
def test_permutation_bit_exact(edp_lib, orc, n):
    edp = edp_lib
    cap = max(n, 8)
    ring = _ppo_ring(edp, cap, H=4, W=4, C=1)
    obs = np.zeros((n, 16), np.uint8)
    # two ingests so that the ring wraps when n < cap
    edp.edp_ingest(ring.ctx, cuda(obs), n)
    idx = torch.full((n,), -1, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, n, 42, 3, idx)
    edp.edp_sync(ring.ctx)
    perm = orc.permutation(n, 42, 3)
    slots = np.array([orc.ring_slot(cap, n, int(j)) for j in perm], np.int64)
    assert np.array_equal(to_np(idx), slots)


def test_permutation_after_wrap(edp_lib, orc):
    edp = edp_lib
    cap = 1000
    ring = _ppo_ring(edp, cap, H=4, W=4, C=1)
    obs = np.zeros((cap, 16), np.uint8)
    edp.edp_ingest(ring.ctx, cuda(obs[:700]), 700)
    edp.edp_ingest(ring.ctx, cuda(obs), cap)  # total 1700, oldest slot 700
    idx = torch.full((cap,), -1, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, cap, 5, 0, idx)
    edp.edp_sync(ring.ctx)
    perm = orc.permutation(cap, 5, 0)
    assert np.array_equal(to_np(idx), (700 + perm) % cap)
    with pytest.raises(edp.EdpError):
        edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, cap - 1, 5, 0, idx)


def test_ppo_iteration_full_size(edp_lib, orc):
    """256 envs x 128 steps of uint8 64x64x3 observations: GAE, Philox
    shuffle of 32,768 samples into 8 mini-batches of 4,096, each delivered
    as bf16 [4096, 3, 64, 64] with gathered normalised advantages and
    returns."""
    edp = edp_lib
    T, E, H, W, C = 128, 256, 64, 64, 3
    n, M = T * E, 8
    mb = n // M
    obs, r, v, d = fx.ppo_rollout(2, T, E)
    ring = _ppo_ring(edp, n)
    edp.edp_ingest(ring.ctx, cuda(obs), n)
    adv, ret, nrm = _gae(edp, ring, r, v, d)
    idx = torch.empty(n, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, n, 2, 0, idx)
    ra, rr = orc.gae(r, v, d, G, LAM)
    rn, _, _ = orc.normalize(ra.ravel())
    assert np.abs(to_np(nrm).ravel() - rn).max() <= 1e-5
    perm = orc.permutation(n, 2, 0)
    edp.edp_sync(ring.ctx)
    assert np.array_equal(to_np(idx), perm)  # fresh ring: slot == offset
    nrm_flat, ret_flat = nrm.view(-1), ret.view(-1)
    for m in range(M):
        out = torch.empty((mb, C, H, W), dtype=torch.bfloat16, device="cuda")
        a_out = torch.full((mb,), float("nan"), device="cuda")
        r_out = torch.full((mb,), float("nan"), device="cuda")
        sub = idx[m * mb:(m + 1) * mb]
        edp.edp_deliver(ring.ctx, sub, mb, edp.make_batch(
            out, gather=[(nrm_flat, a_out), (ret_flat, r_out)]))
        edp.edp_sync(ring.ctx)
        # gathered scalars are the GPU's own advantages at the shuffled ids
        j = perm[m * mb:(m + 1) * mb]
        assert np.array_equal(bits(a_out), bits(nrm_flat)[j])
        assert np.array_equal(bits(r_out), bits(ret_flat)[j])
        if m in (0, M - 1):
            ref, _, _ = orc.deliver_ppo(obs, n, n, H, W, C, j, rn.astype(np.float32),
                                        rr.ravel().astype(np.float32))
            assert np.array_equal(bits(out), ref)
        else:  # spot check a stride of samples
            s = np.arange(0, mb, 97)
            ref, _, _ = orc.deliver_ppo(obs, n, n, H, W, C, j[s],
                                        rn.astype(np.float32),
                                        rr.ravel().astype(np.float32))
            assert np.array_equal(bits(out)[s], ref)


@pytest.mark.parametrize("C", [1, 2, 3, 4])
def test_hwc_chw_channels(edp_lib, orc, C):
    edp = edp_lib
    H, W, cap = 8, 16, 50
    rng = np.random.default_rng(C)
    obs = rng.integers(0, 256, size=(cap + 13, H * W * C), dtype=np.uint8)
    ring = _ppo_ring(edp, cap, H=H, W=W, C=C)
    edp.edp_ingest(ring.ctx, cuda(obs[:cap]), cap)
    edp.edp_ingest(ring.ctx, cuda(obs[cap:]), 13)
    o_ring = np.zeros((cap, H * W * C), np.uint8)
    orc.ring_write(o_ring, cap, 0, obs[:cap])
    orc.ring_write(o_ring, cap, cap, obs[cap:])
    B = 77
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 1, 1, idx)
    out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
    edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(out))
    edp.edp_sync(ring.ctx)
    ref_idx = orc.sample_uniform(cap, cap + 13, cap, B, 1, 1)
    assert np.array_equal(to_np(idx), ref_idx)
    dummy = np.zeros(cap, np.float32)
    ref, _, _ = orc.deliver_ppo(o_ring, cap, cap + 13, H, W, C, ref_idx, dummy, dummy)
    assert np.array_equal(bits(out), ref)


def test_ppo_iteration_in_one_call(edp_lib, orc):
    """The whole iteration delivered by one call (granularity g_del = 1),
    with GAE on a second stream beside the shuffle: mini-batch m is rows
    [4096 m, 4096 (m + 1)) of the output and equals, bit for bit, what the
    m-th per-mini-batch call delivers; strided rows equal the oracle."""
    edp = edp_lib
    T, E, H, W, C = 128, 256, 64, 64, 3
    n, M = T * E, 8
    mb = n // M
    obs, r, v, d = fx.ppo_rollout(3, T, E)
    ring = _ppo_ring(edp, n)
    edp.edp_ingest(ring.ctx, cuda(obs), n)
    dr, dv, dd = cuda(r), cuda(v), cuda(d)
    adv = torch.empty((T, E), device="cuda")
    ret = torch.empty((T, E), device="cuda")
    nrm = torch.empty((T, E), device="cuda")
    idx = torch.empty(n, dtype=torch.int64, device="cuda")
    side = torch.cuda.Stream()
    fork, gae_done = torch.cuda.Event(), torch.cuda.Event()
    torch.cuda.synchronize()
    fork.record()
    with torch.cuda.stream(side):
        side.wait_event(fork)
        edp.edp_gae(ring.ctx, dr, dv, dd, T, E, G, LAM, adv, ret, nrm, stream=side)
        gae_done.record()
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, n, 3, 1, idx)
    torch.cuda.current_stream().wait_event(gae_done)
    out = torch.full((n, C, H, W), float("nan"), dtype=torch.bfloat16, device="cuda")
    a_all = torch.full((n,), float("nan"), device="cuda")
    r_all = torch.full((n,), float("nan"), device="cuda")
    nrm_flat, ret_flat = nrm.view(-1), ret.view(-1)
    edp.edp_deliver(ring.ctx, idx, n, edp.make_batch(
        out, gather=[(nrm_flat, a_all), (ret_flat, r_all)]))
    edp.edp_sync(ring.ctx)
    perm = orc.permutation(n, 3, 1)
    assert np.array_equal(to_np(idx), perm)
    ra, rr = orc.gae(r, v, d, G, LAM)
    rn, _, _ = orc.normalize(ra.ravel())
    assert np.abs(to_np(nrm).ravel() - rn).max() <= 1e-5
    assert np.array_equal(bits(a_all), bits(nrm_flat)[perm])
    assert np.array_equal(bits(r_all), bits(ret_flat)[perm])
    full = bits(out)
    for m in (0, 3, M - 1):
        o = torch.empty((mb, C, H, W), dtype=torch.bfloat16, device="cuda")
        edp.edp_deliver(ring.ctx, idx[m * mb:(m + 1) * mb], mb, edp.make_batch(o))
        edp.edp_sync(ring.ctx)
        assert np.array_equal(bits(o), full[m * mb:(m + 1) * mb])
    s = np.arange(0, n, 61)
    ref, _, _ = orc.deliver_ppo(obs, n, n, H, W, C, perm[s], rn.astype(np.float32),
                                rr.ravel().astype(np.float32))
    assert np.array_equal(full[s], ref)
