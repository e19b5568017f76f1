"""Pins of the oracle's prioritized replay (Schaul et al., proportional
variant, stratified): inverse-CDF sampling, importance weights, priority
updates with duplicates, deferred priorities, and the TD-error rule.
"""
import numpy as np
import pytest


@pytest.mark.parametrize("fn", ["scan", "bisect"])
def test_inverse_cdf_exhaustive(orc, fn):
    """With B == S every stratum is one target t = k, so the sampler must
    enumerate the expanded list (slot i repeated q_i times), exhaustively."""
    sample = getattr(orc, "sample_prioritized_" + fn)
    rng = np.random.default_rng(1)
    for cap in range(1, 65):
        q = rng.integers(0, 5, size=cap).astype(np.uint32)
        q[rng.random(cap) < 0.3] = 0
        if q.sum() == 0:
            q[rng.integers(cap)] = 1
        S = int(q.sum())
        idx, qq = sample(q, S, seed=cap, round_=0)
        expected = np.repeat(np.arange(cap), q)
        assert idx.tolist() == expected.tolist()
        assert qq.tolist() == q[expected].tolist()


def test_scan_equals_bisect_large(orc):
    rng = np.random.default_rng(2)
    q = rng.integers(0, 1 << 22, size=100_003).astype(np.uint32)
    q[rng.random(q.size) < 0.2] = 0
    for r in range(3):
        a = orc.sample_prioritized_scan(q, 512, 7, r)
        b = orc.sample_prioritized_bisect(q, 512, 7, r)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
        assert np.all(q[a[0]] > 0)


def test_strata_partition(orc):
    rng = np.random.default_rng(3)
    for S, B in [(1, 1), (7, 3), (1000, 512), (2**52 + 12345, 512), (5, 8)]:
        prev_hi = 0
        for k in range(B):
            lo, hi = (k * S) // B, ((k + 1) * S) // B
            assert lo == prev_hi
            prev_hi = hi
            u = int(rng.integers(0, 2**63)) * 2 + 1
            t = orc.stratum_target(S, B, k, u)
            if hi > lo:
                assert lo <= t < hi
            else:
                assert t == lo
        assert prev_hi == S


def test_sampling_frequencies_chi_square(orc):
    from scipy.stats import chi2
    rng = np.random.default_rng(4)
    q = rng.integers(1, 1000, size=64).astype(np.uint32)
    counts = np.zeros(64)
    B, rounds = 512, 2000
    for r in range(rounds):
        idx, _ = orc.sample_prioritized_bisect(q, B, 11, r)
        counts += np.bincount(idx, minlength=64)
    expected = B * rounds * q / q.sum()
    stat = float(((counts - expected) ** 2 / expected).sum())
    p = float(chi2.sf(stat, 63))
    # stratification makes the counts *less* variable than multinomial, so
    # only the upper tail is a failure
    assert p > 1e-4, (stat, p)


def test_equal_priorities_are_stratified_uniform(orc):
    cap, B = 1000, 100
    q = np.full(cap, 7, np.uint32)
    idx, _ = orc.sample_prioritized_scan(q, B, 3, 0)
    # stratum k covers slots [10k, 10k+10)
    assert np.all(idx // 10 == np.arange(B))


def test_is_weights_closed_forms(orc):
    w = orc.is_weights(np.full(17, 12345, np.uint32), 0.4)
    assert np.all(w == 1.0)
    q = np.array([100, 400, 100, 400, 1600], np.uint32)
    w = orc.is_weights(q, 0.4)
    exp = np.array([(100.0 / x) ** 0.4 for x in q]).astype(np.float32)
    assert np.array_equal(w, exp)
    assert w.max() == 1.0
    # beta = 0: no correction; beta = 1: plain ratio
    assert np.all(orc.is_weights(q, 0.0) == 1.0)
    assert np.array_equal(orc.is_weights(q, 1.0),
                          (100.0 / q.astype(np.float64)).astype(np.float32))


def _model_update(leaves, pending, qmax, cap, total, defer, idx, q):
    size = min(total, cap)
    oldest = (total - size) % cap
    for s, v in zip(idx, q):
        if s < 0 or s >= cap:
            continue
        k = (s - oldest) % cap
        if k >= size:
            continue
        qmax = max(qmax, v)
        if defer and k == size - 1:
            pending = v
        else:
            leaves[s] = v
    return pending, qmax


@pytest.mark.parametrize("defer", [0, 1])
def test_update_last_wins(orc, defer):
    rng = np.random.default_rng(5 + defer)
    cap = 40
    st = orc.PerState(cap, defer)
    total = 0
    leaves = np.zeros(cap, np.uint32)
    pending, qmax = 0, 1 << 20
    for step in range(30):
        n = int(rng.integers(0, 12))
        qi = rng.integers(1, 1 << 24, size=n).astype(np.uint32)
        orc.ingest_leaves(st, total, qi)
        for j in range(n):  # sequential model of insertion
            iid = total + j
            qmax = max(qmax, int(qi[j]))
            if defer:
                if iid >= 1 and cap >= 2:
                    leaves[(iid - 1) % cap] = pending
                leaves[iid % cap] = 0
                pending = int(qi[j])
            else:
                leaves[iid % cap] = qi[j]
        total += n
        m = int(rng.integers(1, 30))
        idx = rng.integers(-2, cap + 3, size=m)
        idx[: m // 2] = idx[0]  # duplicates
        qu = rng.integers(1, 1 << 30, size=m).astype(np.uint32)
        orc.update_leaves(st, total, idx, qu)
        pending, qmax = _model_update(leaves, pending, qmax, cap, total, defer,
                                      idx.tolist(), qu.tolist())
        assert np.array_equal(st.leaves, leaves), step
        assert int(st.pending[0]) == pending
        assert int(st.qmax[0]) == qmax
        if defer and total:
            assert st.leaves[(total - 1) % cap] == 0  # newest never sampleable


def test_default_priority_is_running_max(orc):
    st = orc.PerState(8, 0)
    orc.ingest_leaves_default(st, 0, 3)
    assert st.leaves[:3].tolist() == [1 << 20] * 3
    orc.update_leaves(st, 3, np.array([1]), np.array([5 << 20], np.uint32))
    orc.ingest_leaves_default(st, 3, 2)
    assert st.leaves[3:5].tolist() == [5 << 20] * 2


def test_priority_from_td(orc):
    rng = np.random.default_rng(6)
    td = rng.exponential(1.0, 100_000).astype(np.float32)
    td[:5] = [0.0, -2.5, 1e-30, 1e6, 3.0]
    q = orc.priorities_from_td(td, 0.6, 1e-6)
    ref = np.rint((np.abs(td.astype(np.float64)) + 1e-6) ** 0.6 * 2.0**20)
    ref = np.clip(ref, 1, 2**32 - 1).astype(np.uint32)
    assert np.array_equal(q, ref)
    # both ends of the clamp to [1, 2^32 - 1]: a zero error without eps, and
    # errors whose priority exceeds 32 bits
    q0 = orc.priorities_from_td(np.array([0.0, 1e9, -1e9], np.float32), 0.6, 0.0)
    assert q0.tolist() == [1, 2**32 - 1, 2**32 - 1]
