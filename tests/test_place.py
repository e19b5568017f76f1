"""The library's placement scan (edp_place_choose, edp_place_map) against
the oracle's restatement of Sec. 5.1-5.2 and Alg. 1, on random options;
invalid options are rejected.  Host-only calls: these run without a GPU."""
import math
import random

import pytest

from oracle import place
from paper_2609_24456_gb300 import edp

GB = 1e9


@pytest.fixture(scope="module", autouse=True)
def _library():
    """Build and load libedp (nvcc cross-compiles; no GPU is needed)."""
    from paper_2609_24456_gb300 import build
    build.build()
    edp.lib()


def _random_options(rng):
    opts = []
    for _ in range(rng.randint(1, 5)):
        o = dict(bw_in=rng.uniform(1, 100) * GB, bw_out=rng.uniform(1, 7000) * GB,
                 mem=rng.uniform(0, 500) * GB)
        if rng.random() < 0.4:
            o.update(bw_out2=rng.uniform(1, 300) * GB, mem2=rng.uniform(0, 500) * GB)
        opts.append(o)
    return opts


def test_choice_and_latencies_match_the_oracle():
    rng = random.Random(9)
    for _ in range(300):
        opts = _random_options(rng)
        c, x = rng.uniform(1e4, 2e6), rng.uniform(1e2, 1e6)
        got, ts = edp.edp_place_choose(opts, c, x)
        ref, ref_ts = place.choose(opts, c, x)
        assert got == ref
        assert ts == ref_ts  # same operations in the same order
        xs = [rng.uniform(1e2, 1e6) for _ in range(20)]
        assert edp.edp_place_map(opts, c, xs) == place.placement_map(opts, c, xs)


@pytest.mark.parametrize("bad", [dict(bw_in=0.0), dict(bw_out=-1.0), dict(mem=-1.0),
                                 dict(bw_out=math.inf), dict(bw_out2=0.0, mem2=1.0)])
def test_invalid_options_are_rejected(bad):
    o = dict(bw_in=1 * GB, bw_out=1 * GB, mem=1 * GB)
    o.update(bad)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_place_choose([o], 10, 1.0)
    assert e.value.status == edp.EDP_ERR_INVALID


def test_invalid_sizes_are_rejected():
    o = [dict(bw_in=1 * GB, bw_out=1 * GB, mem=1 * GB)]
    for c, x in [(0.0, 1.0), (1.0, 0.0), (math.nan, 1.0), (1.0, -3.0)]:
        with pytest.raises(edp.EdpError):
            edp.edp_place_choose(o, c, x)
    with pytest.raises(edp.EdpError):
        edp.edp_place_map(o, 10, [1.0, 0.0])
