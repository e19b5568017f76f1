"""Pins of the placement model (Sec. 5.1-5.2, Eq. 1, Alg. 1) against values
worked out by hand and against brute force."""
import math
import random

from oracle import place

GB = 1e9
HOST = dict(bw_in=50 * GB, bw_out=10 * GB, mem=1000 * GB)      # slow, large
PINNED = dict(bw_in=40 * GB, bw_out=200 * GB, mem=200 * GB)
HBM = dict(bw_in=200 * GB, bw_out=6000 * GB, mem=250 * GB)     # fast, small
SPLIT = dict(bw_in=200 * GB, bw_out=6000 * GB, mem=250 * GB,
             bw_out2=200 * GB, mem2=200 * GB)


def test_two_legs():
    # x = 1 MB: 1e6/50e9 + 1e6/10e9 = 20 us + 100 us
    assert math.isclose(place.transfer_latency(HOST, 1, 1e6), 120e-6, rel_tol=1e-15)


def test_capacity_constraint():
    # C_buf x = 1e6 * 300e3 = 300 GB > 250 GB of HBM
    assert place.transfer_latency(HBM, 1e6, 300e3) == math.inf
    assert place.transfer_latency(HBM, 1e6, 250e3) < math.inf  # exactly fits


def test_two_tier_mixture():
    # C_buf x = 500 GB > 450 GB: infeasible; 300 GB: h = 250/300
    assert place.transfer_latency(SPLIT, 1e6, 500e3) == math.inf
    x = 300e3
    h = 250 / 300
    want = x / (200 * GB) + x * (h / (6000 * GB) + (1 - h) / (200 * GB))
    assert math.isclose(place.transfer_latency(SPLIT, 1e6, x), want, rel_tol=1e-15)
    # everything fits in tier 1: the same as the single-tier HBM option
    assert place.transfer_latency(SPLIT, 1e6, 100e3) == place.transfer_latency(HBM, 1e6, 100e3)


def test_scan_follows_the_regimes():
    opts = [HOST, PINNED, HBM, SPLIT]
    c = 1e6
    # bandwidth-dominated: everything fits, HBM is fastest (first of the tie
    # HBM / SPLIT-with-h=1 wins)
    assert place.choose(opts, c, 10e3)[0] == 2
    # HBM full: the split keeps most reads in HBM
    assert place.choose(opts, c, 300e3)[0] == 3
    # only the host holds it
    assert place.choose(opts, c, 800e3)[0] == 0
    # nothing holds it
    assert place.choose(opts, c, 2e6)[0] == 4
    assert place.placement_map(opts, c, [10e3, 300e3, 800e3, 2e6]) == [2, 3, 0, 4]


def test_scan_is_the_brute_force_minimum():
    rng = random.Random(5)
    for _ in range(300):
        opts = []
        for _ in range(rng.randint(1, 5)):
            o = dict(bw_in=rng.uniform(1, 100) * GB, bw_out=rng.uniform(1, 7000) * GB,
                     mem=rng.uniform(0, 500) * GB)
            if rng.random() < 0.4:
                o.update(bw_out2=rng.uniform(1, 300) * GB, mem2=rng.uniform(0, 500) * GB)
            opts.append(o)
        c, x = rng.uniform(1e4, 2e6), rng.uniform(1e2, 1e6)
        best, ts = place.choose(opts, c, x)
        feasible = [i for i, t in enumerate(ts) if t < math.inf]
        if not feasible:
            assert best == len(opts)
        else:
            assert best == min(feasible, key=lambda i: (ts[i], i))
