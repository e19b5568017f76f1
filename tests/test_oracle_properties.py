"""Invariants of the oracle that hold at any size, checked on generated
cases (hypothesis, derandomised so every run sees the same examples):

- the inverse CDF found by a linear scan equals the one found by bisection
  of the prefix sums, for any leaves (zeros included), batch, seed, round;
- each stratified target lies in its stratum [floor(kS/B), floor((k+1)S/B));
- ring slot and logical offset are inverse maps;
- the two-tier map places every retained id in exactly one slot of one
  tier, no two retained ids in the same slot, and nothing else;
- group-relative advantages are centred within each group.
"""
import numpy as np
import pytest

from hypothesis import given, settings, strategies as st

from oracle import llm

SETTINGS = settings(max_examples=60, derandomize=True, deadline=None)


@SETTINGS
@given(leaves=st.lists(st.integers(0, 2**32 - 1), min_size=1, max_size=200),
       B=st.integers(1, 64), seed=st.integers(0, 2**64 - 1), rnd=st.integers(0, 2**40))
def test_scan_equals_bisect(orc, leaves, B, seed, rnd):
    q = np.array(leaves, np.uint32)
    if int(q.astype(np.uint64).sum()) == 0:
        with pytest.raises(ValueError):
            orc.sample_prioritized_scan(q, B, seed, rnd)
        return
    i1, q1 = orc.sample_prioritized_scan(q, B, seed, rnd)
    i2, q2 = orc.sample_prioritized_bisect(q, B, seed, rnd)
    assert np.array_equal(i1, i2) and np.array_equal(q1, q2)
    assert (q[i1] > 0).all()  # a zero-priority slot is never drawn
    assert np.array_equal(q1, q[i1])


@SETTINGS
@given(S=st.integers(1, 2**64 - 1), B=st.integers(1, 2048), u=st.lists(
    st.integers(0, 2**64 - 1), min_size=3, max_size=3))
def test_strata_hold_their_targets(orc, S, B, u):
    for k in (0, B // 2, B - 1):
        lo, hi = k * S // B, (k + 1) * S // B
        t = orc.stratum_target(S, B, k, u[k % 3])
        assert (lo <= t < hi) if hi > lo else t == lo


@SETTINGS
@given(cap=st.integers(1, 10**6), total=st.integers(0, 10**7), k=st.integers(0, 10**6))
def test_slot_and_offset_are_inverse(orc, cap, total, k):
    size = min(total, cap)
    if size == 0:
        return
    k %= size
    s = orc.ring_slot(cap, total, k)
    assert 0 <= s < cap
    assert orc.ring_offset(cap, total, s) == k


@SETTINGS
@given(cap_h=st.integers(1, 40), cap_c=st.integers(0, 40), total=st.integers(0, 300))
def test_tier_map_is_a_placement(orc, cap_h, cap_c, total):
    cap = cap_h + cap_c
    used = set()
    for L in range(max(0, total - cap - 5), total + 3):
        tier, slot = orc.tier_of(cap, cap_h, total, L)
        retained = total - min(total, cap) <= L < total
        assert (tier >= 0) == retained, (L, tier)
        if tier < 0:
            continue
        assert slot < (cap_h if tier == 0 else cap_c)
        assert (tier, slot) not in used
        used.add((tier, slot))
        # the newest ids fill HBM first
        assert tier == (0 if L >= total - min(total, cap_h) else 1)


@SETTINGS
@given(sizes=st.lists(st.integers(0, 30), min_size=1, max_size=12),
       seed=st.integers(0, 2**32 - 1))
def test_grpo_is_centred(sizes, seed):
    off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.uint64)
    r = np.random.default_rng(seed).standard_normal(int(off[-1])).astype(np.float32) * 3
    a = llm.grpo_advantage(r, off, 1e-6)
    for g in range(len(sizes)):
        seg = a[int(off[g]):int(off[g + 1])].astype(np.float64)
        if len(seg):
            assert abs(seg.sum()) <= 1e-5 * len(seg)
