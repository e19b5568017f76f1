"""Pins of the scheduling model (Sec. 6.2-6.3, Eq. 2, Appendix E) against
values worked out by hand from the formulas, and against properties that
any correct enumeration has."""
import itertools
import random

import pytest

from oracle import sched


def test_inline_timing_is_the_plain_sum():
    # no overlap: T_iter = T_rollout + T_ing(g)/g + T_update + T_del(g)/g
    a, b, t = sched.iter_time(10.0, 20.0, 1.0, 1.0, 0, 2.0, 6.0, 0, 1.0, 5.0)
    assert (a, b, t) == (13.0, 25.0, 38.0)


def test_batched_overlap_hides_the_shorter_side():
    # g >= 1: gamma = 1; hide = min(T_update, Tbar); here Tbar = 8/4 = 2 < 20
    # -> delivery path = 20 + 2 + (0.5 - 2) = 20.5
    assert sched.path_time(20.0, 4.0, 8.0, 0.5, 1) == 20.5
    # the operator is longer than the update: only T_update is hidden
    # Tbar = 30, hide = 20 -> 20 + 30 + 0.5 - 20 = 30.5
    assert sched.path_time(20.0, 1.0, 30.0, 0.5, 1) == 30.5


def test_fractional_overlap_hides_one_minus_g():
    # g = 1/4: gamma = 3/4; Tbar = 2 / 0.25 = 8; hide = 0.75 * min(20, 8) = 6
    # -> 20 + 8 + (1 - 6) = 23
    assert sched.gamma(0.25) == 0.75
    assert sched.path_time(20.0, 0.25, 2.0, 1.0, 1) == 23.0
    # g = 1 is batched, not fractional: gamma = 1
    assert sched.gamma(1.0) == 1.0


def test_overlap_chosen_only_when_sync_is_below_hide():
    # one candidate each; hide_del = min(20, 5) = 5
    for sync, want in [(4.9, 1), (5.1, 0)]:
        best, _ = sched.choose(10.0, 20.0, 100.0, sync, [1.0], [3.0], [1.0], [5.0])
        assert best[1] == want, sync
        assert best[0] == 0  # ingestion overlap would cost 100 - 3


def test_contention_scales_only_the_hidden_part():
    # the fractional example above with half of the hidden time lost:
    # hide = 0.5 * 6 = 3 -> 20 + 8 + 1 - 3 = 26; full contention = inline + sync
    assert sched.path_time(20.0, 0.25, 2.0, 1.0, 1, 0.5) == 26.0
    assert sched.path_time(20.0, 0.25, 2.0, 1.0, 1, 1.0) == 29.0
    assert sched.path_time(20.0, 0.25, 2.0, 1.0, 0, 1.0) == 28.0
    best, _ = sched.choose(0.0, 20.0, 0.0, 1.0, [1.0], [1.0], [0.25], [2.0], 0.0, 1.0)
    assert best[1] == 0  # nothing left to hide: overlap only adds sync


def test_tie_keeps_the_first_candidate():
    # sync == hide: overlapping changes nothing -> inline (0) is kept
    best, _ = sched.choose(10.0, 20.0, 3.0, 5.0, [1.0], [3.0], [1.0], [5.0])
    assert best[:2] == (0, 0)
    # equal per-unit costs at two granularities -> the first index is kept
    best, _ = sched.choose(0.0, 0.0, 0.0, 0.0, [1.0, 2.0], [4.0, 8.0], [1.0], [1.0])
    assert best[2] == 0


def test_choice_is_the_brute_force_minimum_and_decomposes():
    rng = random.Random(7)
    for _ in range(200):
        ni, nd = rng.randint(1, 4), rng.randint(1, 5)
        gi = [rng.choice([0.125, 0.25, 0.5, 1, 2, 4]) for _ in range(ni)]
        gd = [rng.choice([0.125, 0.25, 0.5, 1, 2, 4]) for _ in range(nd)]
        ti = [rng.uniform(0, 50) for _ in range(ni)]
        td = [rng.uniform(0, 50) for _ in range(nd)]
        tr, tu, si, sd = (rng.uniform(0, 40) for _ in range(4))
        best, scores = sched.choose(tr, tu, si, sd, gi, ti, gd, td)
        assert len(scores) == 4 * ni * nd
        assert best[-1] == min(scores)
        # the two paths are independent: best = best ingestion + best delivery
        ing = min(sched.path_time(tr, gi[i], ti[i], si, o)
                  for o, i in itertools.product((0, 1), range(ni)))
        dl = min(sched.path_time(tu, gd[j], td[j], sd, o)
                 for o, j in itertools.product((0, 1), range(nd)))
        assert best[-1] == pytest.approx(ing + dl, rel=1e-12)


def test_candidate_sets():
    assert sched.granularities(True, 8) == [0.125, 0.25, 0.5, 1.0]
    assert sched.granularities(True, 6) == [1 / 6, 2 / 6, 3 / 6, 1.0]
    assert sched.granularities(False, 8) == [1.0, 2.0, 4.0, 8.0]
    assert sched.granularities(False, 5) == [1.0, 2.0, 4.0]
    assert sched.granularities(True, 0) == []
