"""Pins of the oracle's GAE (Schulman et al.) and advantage normalisation:
closed forms, special cases, the recursive form, and numpy statistics."""
import numpy as np

G, LAM = 0.99, 0.95


def _rollout(T, E, seed, done_p=0.05):
    rng = np.random.default_rng(seed)
    r = rng.standard_normal((T, E)).astype(np.float32)
    v = rng.standard_normal((T + 1, E)).astype(np.float32)
    d = (rng.random((T, E)) < done_p).astype(np.uint8)
    return r, v, d


def test_constant_reward_closed_form(orc):
    T, E, c, val = 128, 3, 0.5, 2.0
    r = np.full((T, E), c, np.float32)
    v = np.full((T + 1, E), val, np.float32)
    d = np.zeros((T, E), np.uint8)
    adv, ret = orc.gae(r, v, d, G, LAM)
    t = np.arange(T)[:, None]
    exp = (c + G * val - val) * (1 - (G * LAM) ** (T - t)) / (1 - G * LAM)
    assert np.allclose(adv, exp, rtol=0, atol=1e-12)
    assert np.allclose(ret, exp + val, rtol=0, atol=1e-12)


def test_lambda_zero_is_td_error(orc):
    r, v, d = _rollout(50, 7, 1)
    adv, _ = orc.gae(r, v, d, G, 0.0)
    r64, v64 = r.astype(np.float64), v.astype(np.float64)
    delta = r64 + G * v64[1:] * (1 - d) - v64[:-1]
    assert np.allclose(adv, delta, rtol=0, atol=1e-13)


def test_lambda_one_is_discounted_return(orc):
    r, v, _ = _rollout(40, 5, 2)
    d = np.zeros_like(r, dtype=np.uint8)
    adv, _ = orc.gae(r, v, d, G, 1.0)
    r64, v64 = r.astype(np.float64), v.astype(np.float64)
    T = r.shape[0]
    for t in range(T):
        disc = G ** np.arange(T - t)[:, None]
        ret = (disc * r64[t:]).sum(0) + G ** (T - t) * v64[T]
        assert np.allclose(adv[t], ret - v64[t], rtol=0, atol=1e-11)


def test_done_isolates_segments(orc):
    r, v, d = _rollout(60, 4, 3, done_p=0.0)
    d[20, :] = 1
    a1, _ = orc.gae(r, v, d, G, LAM)
    r2 = r.copy()
    r2[21:] += 5.0
    v2 = v.copy()
    v2[21:] -= 3.0
    a2, _ = orc.gae(r2, v2, d, G, LAM)
    assert np.array_equal(a1[:21], a2[:21])


def test_recursive_form(orc):
    r, v, d = _rollout(130, 9, 4, done_p=0.02)
    adv, ret = orc.gae(r, v, d, G, LAM)
    T, E = r.shape
    A = np.zeros(E)
    for t in range(T - 1, -1, -1):
        nd = 1.0 - d[t]
        delta = r[t] + G * v[t + 1].astype(np.float64) * nd - v[t]
        A = delta + G * LAM * nd * A
        assert np.allclose(adv[t], A, rtol=0, atol=1e-10)
    assert np.allclose(ret, adv + v[:-1], rtol=0, atol=1e-12)


def test_normalize_matches_numpy(orc):
    a = np.random.default_rng(5).standard_normal(32768) * 4 + 1
    out, m, s = orc.normalize(a)
    assert np.isclose(m, a.mean(), rtol=0, atol=1e-12)
    assert np.isclose(s, a.std(ddof=1), rtol=1e-12)
    ref = (a - a.mean()) / (a.std(ddof=1) + 1e-8)
    assert np.allclose(out, ref, rtol=0, atol=1e-12)
    # the 1e-8 sits in the denominator: it is visible at a small spread
    b = np.random.default_rng(6).standard_normal(4096) * 1e-6
    outb, _, _ = orc.normalize(b)
    assert np.allclose(outb, (b - b.mean()) / (b.std(ddof=1) + 1e-8), rtol=1e-12, atol=0)


def test_normalize_constant_rollout_is_zero(orc):
    # zero spread: the advantages are all equal and normalise to 0, not NaN
    out, m, s = orc.normalize(np.full(1024, 0.5))
    assert m == 0.5 and s == 0.0
    assert np.array_equal(out, np.zeros(1024))
