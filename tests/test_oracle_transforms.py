"""Pins of the oracle's byte -> float transforms (exhaustive over bytes)."""
from fractions import Fraction

import numpy as np

MEANS = (0.485, 0.456, 0.406)
STDS = (0.229, 0.224, 0.225)


def test_unit_f32_is_correctly_rounded(orc):
    for b in range(256):
        x = orc.unit_f32(b)
        # IEEE binary32 division by numpy
        assert x == np.float32(b) / np.float32(255)
        # and by exact rationals: within half an ulp of b/255
        if b:
            ulp = np.spacing(np.float32(x))
            assert abs(Fraction(float(x)) - Fraction(b, 255)) <= Fraction(float(ulp)) / 2


def test_bf16_rne_matches_torch(orc):
    import torch
    rng = np.random.default_rng(7)
    xs = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * 3,
        np.array([orc.unit_f32(b) for b in range(256)], np.float32),
        np.array([0.0, -0.0, 1.0, 65504.0, 1e-40, 3.0e38], np.float32),
    ])
    ref = torch.from_numpy(xs).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = np.array([orc.bf16_rne(x) for x in xs], np.uint16)
    assert np.array_equal(got, ref)


def test_bf16_ties_go_to_even(orc):
    # 1 + 2^-8 is halfway between bf16 1.0 and 1.0078125: even is 1.0
    assert orc.bf16_rne(np.float32(1.0 + 2.0**-8)) == 0x3F80
    # 1 + 3*2^-8 is halfway between 1.0078125 (odd) and 1.015625: up
    assert orc.bf16_rne(np.float32(1.0 + 3 * 2.0**-8)) == 0x3F82


def test_norm_bf16_exhaustive(orc):
    import torch
    for c in range(3):
        m, s = np.float32(MEANS[c]), np.float32(STDS[c])
        b = np.arange(256)
        x = b.astype(np.float32) / np.float32(255)
        y = (x - m) / s  # float32 ops, each correctly rounded
        ref = torch.from_numpy(y.astype(np.float32)).to(torch.bfloat16).view(
            torch.int16).numpy().view(np.uint16)
        got = np.array([orc.norm_bf16(v, m, s) for v in range(256)], np.uint16)
        assert np.array_equal(got, ref)


def test_hwc_to_chw_ramp(orc):
    H, W, C = 64, 64, 3
    y, x, c = np.meshgrid(np.arange(H), np.arange(W), np.arange(C), indexing="ij")
    img = (((y * 64 + x) * 3 + c) % 251).astype(np.uint8)
    out = orc.hwc_to_chw_bf16(img)
    lut = np.array([orc.bf16_rne(orc.unit_f32(b)) for b in range(256)], np.uint16)
    assert np.array_equal(out, lut[img.transpose(2, 0, 1)])


def test_norm_chw_matches_per_element(orc):
    rng = np.random.default_rng(8)
    img = rng.integers(0, 256, size=(3, 16, 16), dtype=np.uint8)
    out = orc.norm_chw_bf16(img, MEANS, STDS)
    for c in range(3):
        lut = np.array([orc.norm_bf16(b, MEANS[c], STDS[c]) for b in range(256)],
                       np.uint16)
        assert np.array_equal(out[c], lut[img[c]])


def _bf16(x):
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(
        torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def test_deliver_ppo_scalars_follow_logical_offset(orc):
    # a wrapped ring: ids 5..12 in 8 slots, id L in slot L mod 8; a sample's
    # advantage and return are those of its logical offset (its position
    # from the oldest stored transition), its image the slot's, CHW
    H, W, Cc, cap, total = 2, 3, 3, 8, 13
    rng = np.random.default_rng(11)
    ring = rng.integers(0, 256, (cap, H * W * Cc), dtype=np.uint8)
    ids = list(range(total - cap, total))
    adv = np.arange(cap, dtype=np.float32) + 100
    ret = -np.arange(cap, dtype=np.float32)
    idx = np.array([0, 4, 5, 7, 4, 2], np.int64)
    out, a, r = orc.deliver_ppo(ring, cap, total, H, W, Cc, idx, adv, ret)
    for b, s in enumerate(idx):
        k = [L % cap for L in ids].index(s)
        assert a[b] == 100 + k and r[b] == -k
        img = ring[s].reshape(H, W, Cc).transpose(2, 0, 1).astype(np.float32) / np.float32(255)
        assert np.array_equal(out[b], _bf16(img))


def test_deliver_mm_collates(orc):
    Cc, HW, L, cap = 3, 10, 5, 7
    rng = np.random.default_rng(12)
    ring = rng.integers(0, 256, (cap, Cc * HW), dtype=np.uint8)
    tok = rng.integers(0, 32000, (cap, L), dtype=np.int32)
    rew = rng.standard_normal(cap).astype(np.float32)
    idx = np.array([6, 0, 3, 3, 1], np.int64)
    m = np.array(MEANS, np.float32)
    sd = np.array(STDS, np.float32)
    out, t, r = orc.deliver_mm(ring, tok, rew, Cc, HW, idx, m, sd)
    assert np.array_equal(t, tok[idx])
    assert np.array_equal(r, rew[idx])
    x = ring[idx].reshape(len(idx), Cc, HW).astype(np.float32) / np.float32(255)
    y = (x - m[None, :, None]) / sd[None, :, None]
    assert np.array_equal(out.reshape(len(idx), Cc, HW), _bf16(y))
