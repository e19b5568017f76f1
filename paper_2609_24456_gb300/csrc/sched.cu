// sched.cu -- latency-aware scheduling of ingestion and delivery (Sec. 6):
// the iteration-latency model (Sec. 6.2, Appendix E) and the cost-based
// choice of timing and granularity (Eq. 2, Sec. 6.3).  Host code only; the
// formulas are stated in edp.h.
#include <cmath>

#include "edp_internal.cuh"

namespace {

bool finite_nonneg(double x) { return std::isfinite(x) && x >= 0.0; }
bool finite_pos(double x) { return std::isfinite(x) && x > 0.0; }

// one operator path:
//   T_neighbour + Tbar(g) + o (T_sync - (1 - c) gamma(g) min(T_neighbour, Tbar(g)))
double path(double t_neighbour, double g, double t_op, double t_sync, double c,
            uint32_t overlap) {
  const double tbar = t_op / g;
  if (!overlap) return t_neighbour + tbar;
  const double gamma = g >= 1.0 ? 1.0 : 1.0 - g;
  const double hide = (1.0 - c) * (gamma * (t_neighbour < tbar ? t_neighbour : tbar));
  return t_neighbour + tbar + (t_sync - hide);
}

bool unit_interval(double x) { return std::isfinite(x) && x >= 0.0 && x <= 1.0; }

}  // namespace

extern "C" {

edp_status edp_sched_choose(const edp_sched_costs *c, edp_sched_choice *best,
                            double *t_iter_all) {
  if (!c || !best || !c->g_ing || !c->t_ing || !c->g_del || !c->t_del ||
      c->n_ing == 0 || c->n_del == 0)
    return EDP_ERR_INVALID;
  if (!finite_nonneg(c->t_rollout) || !finite_nonneg(c->t_update) ||
      !finite_nonneg(c->t_sync_ing) || !finite_nonneg(c->t_sync_del) ||
      !unit_interval(c->contention_ing) || !unit_interval(c->contention_del))
    return EDP_ERR_INVALID;
  for (uint32_t i = 0; i < c->n_ing; ++i)
    if (!finite_pos(c->g_ing[i]) || !finite_nonneg(c->t_ing[i])) return EDP_ERR_INVALID;
  for (uint32_t i = 0; i < c->n_del; ++i)
    if (!finite_pos(c->g_del[i]) || !finite_nonneg(c->t_del[i])) return EDP_ERR_INVALID;
  bool have = false;
  edp_sched_choice b{};
  uint64_t k = 0;
  for (uint32_t oi = 0; oi < 2; ++oi)
    for (uint32_t od = 0; od < 2; ++od)
      for (uint32_t ii = 0; ii < c->n_ing; ++ii)
        for (uint32_t id = 0; id < c->n_del; ++id, ++k) {
          const double ti = path(c->t_rollout, c->g_ing[ii], c->t_ing[ii], c->t_sync_ing,
                                 c->contention_ing, oi);
          const double td = path(c->t_update, c->g_del[id], c->t_del[id], c->t_sync_del,
                                 c->contention_del, od);
          const double t = ti + td;
          if (t_iter_all) t_iter_all[k] = t;
          if (!have || t < b.t_iter) {
            have = true;
            b.overlap_ing = oi;
            b.overlap_del = od;
            b.i_ing = ii;
            b.i_del = id;
            b.g_ing = c->g_ing[ii];
            b.g_del = c->g_del[id];
            b.t_ing_path = ti;
            b.t_del_path = td;
            b.t_iter = t;
          }
        }
  *best = b;
  return EDP_OK;
}

uint32_t edp_sched_granularities(uint32_t on_policy, uint32_t m, double *g, uint32_t cap) {
  if (m == 0) return 0;
  uint32_t n = 0;
  if (on_policy) {
    for (uint32_t k = 1; k <= m; ++k)
      if (m % k == 0) {
        if (g && n < cap) g[n] = (double)k / (double)m;
        ++n;
      }
  } else {
    for (uint64_t k = 1; k <= m; k *= 2) {
      if (g && n < cap) g[n] = (double)k;
      ++n;
    }
  }
  return n;
}

}  // extern "C"
