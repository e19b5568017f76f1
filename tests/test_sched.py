"""The library's scheduler (edp_sched_choose, edp_sched_granularities)
against the oracle's restatement of Sec. 6.2-6.3: same choice and the same
score for every candidate, on random costs; invalid costs are rejected.
Host-only calls: these run without a GPU."""
import math
import random

import pytest

from oracle import sched
from paper_2609_24456_gb300 import edp



@pytest.fixture(scope="module", autouse=True)
def _library():
    """Build and load libedp (nvcc cross-compiles; no GPU is needed)."""
    from paper_2609_24456_gb300 import build
    build.build()
    edp.lib()


def _random_costs(rng):
    ni, nd = rng.randint(1, 4), rng.randint(1, 6)
    pick = lambda: rng.choice([1 / 8, 1 / 4, 1 / 2, 1.0, 2.0, 4.0, 8.0])
    gi = [pick() for _ in range(ni)]
    gd = [pick() for _ in range(nd)]
    ti = [rng.uniform(0, 500) for _ in range(ni)]
    td = [rng.uniform(0, 500) for _ in range(nd)]
    tr, tu, si, sd = (rng.uniform(0, 300) for _ in range(4))
    return tr, tu, si, sd, gi, ti, gd, td, rng.choice([0.0, rng.random()]), rng.random()


def test_choice_and_scores_match_the_oracle():
    rng = random.Random(11)
    for _ in range(300):
        *args, ci, cd = _random_costs(rng)
        got, scores = edp.edp_sched_choose(*args, all_scores=True, contention_ing=ci,
                                           contention_del=cd)
        best, ref_scores = sched.choose(*args, ci, cd)
        assert scores == ref_scores  # same operations in the same order
        o_ing, o_del, i, j, a, b, t = best
        assert (got.overlap_ing, got.overlap_del, got.i_ing, got.i_del) == (o_ing, o_del, i, j)
        assert (got.t_ing_path, got.t_del_path, got.t_iter) == (a, b, t)
        assert got.g_ing == args[4][i] and got.g_del == args[6][j]


@pytest.mark.parametrize("on_policy,m", [(True, 8), (True, 12), (True, 1), (False, 1),
                                         (False, 16), (False, 100), (True, 0)])
def test_granularities_match_the_oracle(on_policy, m):
    assert edp.edp_sched_granularities(on_policy, m) == sched.granularities(on_policy, m)


@pytest.mark.parametrize("bad", [
    dict(g_ing=[0.0]), dict(g_del=[-1.0]), dict(t_del=[math.nan]),
    dict(t_ing=[-0.1]), dict(t_update=math.inf), dict(t_sync_del=-1.0),
    dict(g_ing=[], t_ing=[]), dict(contention_del=1.5), dict(contention_ing=-0.1)])
def test_invalid_costs_are_rejected(bad):
    kw = dict(t_rollout=1.0, t_update=1.0, t_sync_ing=0.0, t_sync_del=0.0,
              g_ing=[1.0], t_ing=[1.0], g_del=[1.0], t_del=[1.0])
    kw.update(bad)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_sched_choose(**kw)
    assert e.value.status == edp.EDP_ERR_INVALID
