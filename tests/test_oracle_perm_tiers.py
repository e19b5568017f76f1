"""Pins of the oracle's on-policy shuffle and two-tier placement map."""
import numpy as np
import pytest


@pytest.mark.parametrize("n", [1, 2, 5, 1000, 32768])
def test_permutation_is_sorted_random_keys(orc, n):
    perm = orc.permutation(n, 123, 4)
    assert np.array_equal(np.sort(perm), np.arange(n))  # bijection
    keys = np.array([orc.philox_u64(123, j, 4, 2) for j in range(n)],
                    dtype=np.uint64)
    ref = np.lexsort((np.arange(n), keys))  # numpy: by key, then index
    assert len(np.unique(keys)) == n  # so the index tie-break never decides
    assert np.array_equal(perm, ref)


def test_minibatches_partition_rollout(orc):
    n, M = 32768, 8
    perm = orc.permutation(n, 9, 0)
    parts = [perm[m * (n // M):(m + 1) * (n // M)] for m in range(M)]
    seen = np.concatenate(parts)
    assert len(np.unique(seen)) == n
    assert all(len(p) == n // M for p in parts)
    # a new iteration reshuffles
    assert not np.array_equal(perm, orc.permutation(n, 9, 1))


def test_tier_map_against_physical_simulation(orc):
    """Simulate two physical rings, one insertion at a time: a new
    transition enters HBM; when HBM is full its oldest entry first moves to
    the host ring, whose oldest entry is evicted when it is full.  Check the
    arithmetic map against where each id physically is."""
    rng = np.random.default_rng(12)
    for cap_h, cap_c in [(1, 1), (3, 2), (4, 7), (8, 8), (5, 13)]:
        cap = cap_h + cap_c
        hbm, host = [], []  # logical ids, oldest first
        total = 0
        for step in range(25 + 2 * cap):
            # one at a time while the tiers fill (HBM partly full, then the
            # host tier), then random batches
            n = 1 if step < 2 * cap else int(rng.integers(0, cap + 1))
            for j in range(n):
                if len(hbm) == cap_h:
                    if len(host) == cap_c:
                        host.pop(0)
                    host.append(hbm.pop(0))
                hbm.append(total + j)
            total += n
            for L in range(max(0, total - cap - 3), total + 2):
                tier, slot = orc.tier_of(cap, cap_h, total, L)
                if tier == 0:
                    assert L in hbm and slot == L % cap_h
                elif tier == 1:
                    assert L in host and slot == L % cap_c
                else:
                    assert L not in hbm and L not in host
