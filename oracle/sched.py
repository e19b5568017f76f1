"""Latency-aware scheduling, written out from the paper (test infrastructure
only: the tests and the benchmark's CPU leg may use it, the library never).

Sec. 6.2 models one RL iteration as the exposed ingestion path plus the
exposed delivery path; Appendix E gives the hidden terms; Eq. 2 (Sec. 6.3)
picks the timing flags and granularities that minimise the sum by scoring
every candidate.  Plain Python floats, the formulas in the paper's order.
"""


def per_unit(t_of_g, g):
    """Tbar(g) = T(g) / g, the cost of one unit at granularity g (Sec. 6.2)."""
    return t_of_g / g


def gamma(g):
    """Overlapable share (Appendix E): 1 for g >= 1, 1 - g for 0 < g < 1."""
    return 1.0 if g >= 1 else 1.0 - g


def hide(t_neighbour, g, t_of_g, contention=0.0):
    """hide = gamma(g) * min(T_neighbour, Tbar(g)) (Appendix E), where the
    neighbour is the rollout for ingestion and the update for delivery,
    scaled by (1 - contention) -- a factor the paper does not have (it is 0
    there): the share of the overlap lost when operator and neighbour share
    one device."""
    return (1.0 - contention) * (gamma(g) * min(t_neighbour, per_unit(t_of_g, g)))


def path_time(t_neighbour, g, t_of_g, t_sync, overlap, contention=0.0):
    """T_path = T_neighbour + Tbar(g) + overlap * (T_sync - hide) (Sec. 6.2)."""
    t = t_neighbour + per_unit(t_of_g, g)
    if overlap:
        t = t + (t_sync - hide(t_neighbour, g, t_of_g, contention))
    return t


def iter_time(t_rollout, t_update, t_sync_ing, t_sync_del, o_ing, g_ing, t_ing,
              o_del, g_del, t_del, c_ing=0.0, c_del=0.0):
    """T_iter = T_ing-path + T_del-path (Sec. 6.2)."""
    a = path_time(t_rollout, g_ing, t_ing, t_sync_ing, o_ing, c_ing)
    b = path_time(t_update, g_del, t_del, t_sync_del, o_del, c_del)
    return a, b, a + b


def choose(t_rollout, t_update, t_sync_ing, t_sync_del, g_ing, t_ing, g_del, t_del,
           c_ing=0.0, c_del=0.0):
    """Eq. 2: enumerate overlap_ing, overlap_del in {0, 1} and every pair of
    candidate granularities, score each by T_iter, keep the smallest (the
    first one met, in the order o_ing, o_del, i_ing, i_del, on a tie).
    Returns (best tuple, list of all scores in enumeration order)."""
    best, scores = None, []
    for o_ing in (0, 1):
        for o_del in (0, 1):
            for i in range(len(g_ing)):
                for j in range(len(g_del)):
                    a, b, t = iter_time(t_rollout, t_update, t_sync_ing, t_sync_del,
                                        o_ing, g_ing[i], t_ing[i], o_del, g_del[j], t_del[j],
                                        c_ing, c_del)
                    scores.append(t)
                    if best is None or t < best[-1]:
                        best = (o_ing, o_del, i, j, a, b, t)
    return best, scores


def granularities(on_policy, m):
    """Candidate sets (Sec. 6.3): integer batching for off-policy replay (1, 2,
    4, ... up to m), fractional mini-batch steps k/m (k dividing m) for
    on-policy training."""
    if m == 0:
        return []
    if on_policy:
        return [k / m for k in range(1, m + 1) if m % k == 0]
    out, k = [], 1
    while k <= m:
        out.append(float(k))
        k *= 2
    return out
