"""GPU parity of the multimodal payload path through the C ABI: CHW uint8
224x224 images delivered as per-channel normalised bf16 with collated
int32 tokens and rewards, single-tier and two-tier (HBM + page-locked host
memory with demotion), all bit-exact against the oracle."""
import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, fx, to_np

pytestmark = pytest.mark.gpu

MEAN = (0.485, 0.456, 0.406)
STD = (0.229, 0.224, 0.225)
C, H, W, L = 3, 224, 224, 512
F = C * H * W


def _mm_ring(edp, cap, cap_h=None):
    cfg = edp.make_config(cap, (C, H, W), edp.EDP_XFORM_CHW_NORM_BF16,
                          hbm_capacity=cap_h, tokens=L, norm_mean=MEAN,
                          norm_std=STD)
    return edp.Ring(cfg, action=False, done=False)


class Logical:
    """Oracle-side view of the logical ring: slot L mod cap holds id L."""

    def __init__(self, cap, seed):
        self.cap, self.seed, self.total = cap, seed, 0
        self.obs = np.zeros((cap, F), np.uint8)
        self.tok = np.zeros((cap, L), np.int32)
        self.rew = np.zeros(cap, np.float32)

    def ingest(self, orc, n, rew):
        ids = np.arange(self.total, self.total + n)
        orc.ring_write(self.obs, self.cap, self.total, fx.content_bytes(self.seed, ids, F))
        orc.ring_write(self.tok, self.cap, self.total, fx.token_content(self.seed, ids, L))
        orc.ring_write(self.rew, self.cap, self.total, np.ascontiguousarray(rew))
        self.total += n


def _ingest(edp, ring, lg, orc, n, seed, pinned=False):
    obs = torch.empty((n, F), dtype=torch.uint8, device="cuda")
    tok = torch.empty((n, L), dtype=torch.int32, device="cuda")
    fx.content_fill_torch(seed, lg.total, obs)
    fx.token_fill_torch(seed, lg.total, tok)
    _, rew = fx.mm_metadata(seed * 7 + lg.total, n, tokens=0)
    if pinned:
        obs, tok = obs.cpu().pin_memory(), tok.cpu().pin_memory()
    edp.edp_ingest(ring.ctx, obs, n, tokens=tok, reward=cuda(rew))
    lg.ingest(orc, n, rew)


def _deliver_check(edp, orc, ring, lg, B, seed, rnd, subset=None):
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, seed, rnd, idx)
    out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
    tok = torch.full((B, L), -1, dtype=torch.int32, device="cuda")
    rew = torch.full((B,), float("nan"), device="cuda")
    edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(out, tokens=tok, reward=rew))
    edp.edp_sync(ring.ctx)
    size = min(lg.total, lg.cap)
    ref_idx = orc.sample_uniform(lg.cap, lg.total, size, B, seed, rnd)
    assert np.array_equal(to_np(idx), ref_idx)
    sel = np.arange(B) if subset is None else subset
    r_obs, r_tok, r_rew = orc.deliver_mm(lg.obs, lg.tok, lg.rew, C, H * W,
                                         ref_idx[sel], MEAN, STD)
    assert np.array_equal(bits(out).reshape(B, -1)[sel], r_obs)
    assert np.array_equal(to_np(tok)[sel], r_tok)
    assert np.array_equal(bits(rew)[sel], r_rew.view(np.uint32))


def test_mm_single_tier_ragged(edp_lib, orc):
    edp = edp_lib
    cap, seed = 300, 11
    ring = _mm_ring(edp, cap)
    lg = Logical(cap, seed)
    for n in [7, 250, 100, 299]:
        _ingest(edp, ring, lg, orc, n, seed)
        _deliver_check(edp, orc, ring, lg, 101, seed=3, rnd=lg.total)


_RNG_NORM = np.random.default_rng(77)
NORM_CASES = [
    (MEAN, STD, 2),
    # channel 0: mean within an ulp of 143/255, where no (A, B) within 16
    # ulps reproduces the chain for every byte -> the chain is evaluated
    ((0.560784519, 0.456, 0.406), (0.604448199, 0.224, 0.225), 1),
    # a subnormal std: 1/(255 std) overflows -> the chain with IEEE division
    ((0.485, 0.456, 0.406), (1e-40, 0.224, 0.225), 0),
] + [(tuple(_RNG_NORM.uniform(0, 1, 3)), tuple(_RNG_NORM.uniform(0.05, 1.05, 3)), None)
     for _ in range(3)]


@pytest.mark.parametrize("mean,std,path", NORM_CASES)
def test_mm_all_byte_channel_pairs(edp_lib, orc, mean, std, path):
    """All 768 (byte, channel) pairs through the normalisation, bit-exact,
    for each way the kernel evaluates it (one FMA, the chain with a split
    reciprocal, the chain with IEEE division)."""
    edp = edp_lib
    cap = 4
    cfg = edp.make_config(cap, (C, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16,
                          norm_mean=mean, norm_std=std)
    ring = edp.Ring(cfg, action=False, reward=False, done=False)
    if path is not None:
        assert ring.info().norm_path == path
    img = np.tile(np.arange(256, dtype=np.uint8), (cap, C)).reshape(cap, C * 256)
    edp.edp_ingest(ring.ctx, cuda(img), cap)
    idx = torch.arange(cap, dtype=torch.int64, device="cuda")
    out = torch.empty((cap, C, 16, 16), dtype=torch.bfloat16, device="cuda")
    edp.edp_deliver(ring.ctx, idx, cap, edp.make_batch(out))
    edp.edp_sync(ring.ctx)
    for c in range(C):
        lut = np.array([orc.norm_bf16(b, mean[c], std[c]) for b in range(256)],
                       np.uint16)
        assert np.array_equal(bits(out)[:, c].reshape(cap, 256), np.tile(lut, (cap, 1)))


@pytest.mark.parametrize("pinned_src", [False, True])
def test_mm_two_tier(edp_lib, orc, pinned_src):
    edp = edp_lib
    cap, cap_h, seed = 64, 24, 5
    ring = _mm_ring(edp, cap, cap_h)
    lg = Logical(cap, seed)
    for n in [3, 30, 20, 64, 1, 50, 24, 25]:  # includes chunks > cap_h
        _ingest(edp, ring, lg, orc, n, seed, pinned=pinned_src)
        _deliver_check(edp, orc, ring, lg, 40, seed=9, rnd=lg.total)
        # placement: each retained id is in the tier the map says, and
        # nowhere else is read from
        edp.edp_sync(ring.ctx)
        host = ring.host_obs.numpy()
        hbm = ring.obs.cpu().numpy()
        size = min(lg.total, cap)
        for Lid in range(lg.total - size, lg.total):
            tier, slot = orc.tier_of(cap, cap_h, lg.total, Lid)
            row = host[slot] if tier == 1 else hbm[slot]
            assert tier in (0, 1)
            assert np.array_equal(row, lg.obs[Lid % cap]), (Lid, tier)


def test_mm_full_size(edp_lib, orc):
    """200,000 transitions of 3x224x224 images + 512 tokens (~30 GB in HBM),
    batch 1,024: all indices, a subset of delivered samples."""
    edp = edp_lib
    cap, seed, B = 200_000, 1237, 1024
    ring = _mm_ring(edp, cap)
    chunk = 8192
    obs = torch.empty((chunk, F), dtype=torch.uint8, device="cuda")
    tok = torch.empty((chunk, L), dtype=torch.int32, device="cuda")
    _, rew_all = fx.mm_metadata(seed, cap, tokens=0)
    for lo in range(0, cap, chunk):
        n = min(chunk, cap - lo)
        fx.content_fill_torch(seed, lo, obs[:n])
        fx.token_fill_torch(seed, lo, tok[:n])
        edp.edp_ingest(ring.ctx, obs[:n], n, tokens=tok[:n],
                       reward=cuda(rew_all[lo:lo + n]))
    del obs, tok
    for rnd in range(2):
        idx = torch.empty(B, dtype=torch.int64, device="cuda")
        edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 77, rnd, idx)
        out = torch.empty((B, C, H, W), dtype=torch.bfloat16, device="cuda")
        tk = torch.empty((B, L), dtype=torch.int32, device="cuda")
        rw = torch.empty((B,), device="cuda")
        edp.edp_deliver(ring.ctx, idx, B, edp.make_batch(out, tokens=tk, reward=rw))
        edp.edp_sync(ring.ctx)
        ref_idx = orc.sample_uniform(cap, cap, cap, B, 77, rnd)
        assert np.array_equal(to_np(idx), ref_idx)
        sel = np.arange(0, B, 61)
        ids = ref_idx[sel]  # full ring, no wrap: id == slot
        lo_obs = fx.content_bytes(seed, ids, F)
        lo_tok = fx.token_content(seed, ids, L)
        r_obs, r_tok, r_rew = orc.deliver_mm(lo_obs, lo_tok, rew_all[ids], C,
                                             H * W, np.arange(len(sel)), MEAN, STD)
        assert np.array_equal(bits(out).reshape(B, -1)[sel], r_obs)
        assert np.array_equal(to_np(tk)[sel], r_tok)
        assert np.array_equal(bits(rw)[sel], r_rew.view(np.uint32))
