"""Pins of the LLM post-training oracle: group-relative advantages against
values worked out by hand and their invariants, packing against a
hand-built batch."""
import math

import numpy as np

from oracle import llm


def test_grpo_hand_values():
    r = np.array([1, 2, 3, 5, 5, 5, 7, 0, 1], np.float32)
    off = np.array([0, 3, 6, 7, 9], np.uint64)
    a = llm.grpo_advantage(r, off, 0.0)
    # [1,2,3]: mean 2, sample std 1 -> -1, 0, 1; a constant group and a
    # group of one -> 0; [0,1]: mean 0.5, std sqrt(0.5) -> -+0.5/sqrt(0.5)
    h = np.float32(0.5 / math.sqrt(0.5))
    assert list(a) == [-1.0, 0.0, 1.0, 0.0, 0.0, 0.0, 0.0, -h, h]
    # eps enters the denominator only
    a2 = llm.grpo_advantage(r[:3], off[:2], 1.0)
    assert list(a2) == [-0.5, 0.0, 0.5]


def test_grpo_invariants():
    rng = np.random.default_rng(3)
    r = rng.standard_normal(64).astype(np.float32)
    off = np.array([0, 10, 26, 27, 64], np.uint64)
    a = llm.grpo_advantage(r, off, 0.0)
    for g in range(4):
        lo, hi = int(off[g]), int(off[g + 1])
        seg = a[lo:hi].astype(np.float64)
        assert abs(seg.sum()) < 1e-5  # centred
        if hi - lo > 1:  # unit sample variance
            assert abs(seg.var(ddof=1) - 1.0) < 1e-5
    # shift and positive scale of a group's rewards leave A unchanged
    r2 = r.copy()
    r2[10:26] = r2[10:26] * np.float32(4) + np.float32(3)
    b = llm.grpo_advantage(r2, off, 0.0)
    assert np.allclose(a[10:26], b[10:26], atol=1e-6)


def test_pack_hand_batch():
    tok = np.array([10, 11, 12, 20, 30, 31], np.int32)
    off = np.array([0, 3, 4, 6], np.uint64)
    v = np.array([0.5, 1.5, 2.5], np.float32)
    out, ooff, ov = llm.pack(tok, off, [2, 0, 2, 7, 1], v)
    assert list(out) == [30, 31, 10, 11, 12, 30, 31, 20]
    assert list(ooff) == [0, 2, 5, 7, 7, 8]  # index 7 is out of range: empty
    assert list(ov) == [2.5, 2.5, 0.5, 0.5, 0.5, 2.5, 2.5, 1.5]
