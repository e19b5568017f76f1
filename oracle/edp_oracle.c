/*
 * edp_oracle.c -- plain, slow, obviously-correct CPU model of the experience
 * path (ingest, sample, deliver, priority update, GAE, shuffle, tiers).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library path may call, link or
 * load this file; only the test-suite, the smoke check and the benchmark's
 * CPU-baseline leg use it.  It shares no code, header, table or constant
 * generator with the CUDA implementation.
 *
 * The paper (Conduit, "An Experience Data Plane for Distributed RL") stays at
 * the systems level: it names the operators of the experience path --
 * insertion with indices and eviction metadata, sampling, materialisation,
 * concat/reshape, returns/advantages, normalisation, shuffling into
 * mini-batches (Sec. 2.2, "Experience Path Responsibilities") -- and the
 * priority callback of replay (Appendix C, Invariant 2), but never writes out
 * their arithmetic.  Each function below therefore states the published
 * method it follows and the reading it adopts where the text is silent.
 *
 * Floating point is fp64 wherever the definition is real-valued; values that
 * the method itself defines in fp32/bf16 (the byte->float transforms) are
 * computed with one IEEE operation per step, no contraction (built with
 * -ffp-contract=off), so the result is the correctly rounded one.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <math.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_API __attribute__((visibility("default")))

/* Set the threads of the OpenMP loops (timing only; no effect on results). */
ORC_API void orc_set_threads(int n) {
#ifdef _OPENMP
  if (n > 0) omp_set_num_threads(n);
#else
  (void)n;
#endif
}

/* Threads the OpenMP loops over batch rows use (1 without OpenMP). */
ORC_API int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Philox4x32-10, Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As   */
/* Easy as 1, 2, 3" (SC'11): a 4-word counter, a 2-word key, ten rounds.     */
/* Each round multiplies words 0 and 2 by the two round multipliers into     */
/* 64-bit products; the new words are (hi(w2*M1) ^ w1 ^ k0, lo(w2*M1),       */
/* hi(w0*M0) ^ w3 ^ k1, lo(w0*M0)).  The key is advanced by the two Weyl     */
/* constants before every round but the first.                               */
/* ------------------------------------------------------------------------ */
static const uint32_t PHILOX_M0 = 0xD2511F53u;
static const uint32_t PHILOX_M1 = 0xCD9E8D57u;
static const uint32_t PHILOX_W0 = 0x9E3779B9u;
static const uint32_t PHILOX_W1 = 0xBB67AE85u;

ORC_API void orc_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2],
                               uint32_t out[4]) {
  uint32_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint32_t k0 = key[0], k1 = key[1];
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)x0;
    uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)x2;
    uint32_t n0 = (uint32_t)(p1 >> 32) ^ x1 ^ k0;
    uint32_t n1 = (uint32_t)p1;
    uint32_t n2 = (uint32_t)(p0 >> 32) ^ x3 ^ k1;
    uint32_t n3 = (uint32_t)p0;
    x0 = n0; x1 = n1; x2 = n2; x3 = n3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* The 64-bit draw number j of (seed, round, stream): counter =
 * (j, round lo32, stream, round hi32), key = (seed lo32, seed hi32);
 * value = (word1 << 32) | word0.  Streams: 0 uniform sampler, 1 stratified
 * prioritized sampler, 2 shuffle keys. */
ORC_API uint64_t orc_philox_u64(uint64_t seed, uint32_t j, uint64_t round,
                                uint32_t stream) {
  uint32_t c[4] = {j, (uint32_t)round, stream, (uint32_t)(round >> 32)};
  uint32_t k[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t o[4];
  orc_philox4x32_10(c, k, o);
  return ((uint64_t)o[1] << 32) | (uint64_t)o[0];
}

/* floor(a * n / 2^64): maps a uniform 64-bit word onto [0, n). */
ORC_API uint64_t orc_mulhi64(uint64_t a, uint64_t n) {
  unsigned __int128 p = (unsigned __int128)a * (unsigned __int128)n;
  return (uint64_t)(p >> 64);
}

/* ------------------------------------------------------------------------ */
/* Logical ring (Sec. 2.2: off-policy ingestion inserts transitions and      */
/* keeps indices and metadata "for future sampling and eviction").  Reading: */
/* FIFO eviction.  After `total` insertions into `cap` slots the buffer      */
/* holds the newest size = min(total, cap) transitions; logical offset k in  */
/* [0, size) (0 = oldest) lives in slot (total - size + k) mod cap, i.e. the  */
/* transition with logical id L lives in slot L mod cap.                     */
/* ------------------------------------------------------------------------ */
ORC_API uint64_t orc_ring_size(uint64_t cap, uint64_t total) {
  return total < cap ? total : cap;
}

ORC_API uint64_t orc_ring_slot(uint64_t cap, uint64_t total, uint64_t k) {
  uint64_t size = orc_ring_size(cap, total);
  return (total - size + k) % cap;
}

/* logical offset of a slot (inverse of orc_ring_slot) */
ORC_API uint64_t orc_ring_offset(uint64_t cap, uint64_t total, uint64_t slot) {
  uint64_t size = orc_ring_size(cap, total);
  uint64_t oldest = (total - size) % cap;
  return (slot + cap - oldest) % cap;
}

/* Insert n records of rec bytes, one after another, at logical ids
 * total .. total+n-1 of one field of the ring. */
ORC_API void orc_ring_write(uint8_t *ring, uint64_t cap, uint64_t rec,
                            uint64_t total, const uint8_t *src, uint64_t n) {
  for (uint64_t j = 0; j < n; ++j) {
    uint64_t slot = (total + j) % cap;
    memcpy(ring + slot * rec, src + j * rec, rec);
  }
}

/* ------------------------------------------------------------------------ */
/* Priorities (Schaul et al., "Prioritized Experience Replay", ICLR'16; the  */
/* paper's replay-state callback, Appendix C Invariant 2).  Priorities are   */
/* unsigned 32-bit fixed point (1.0 == 2^20).                                */
/*                                                                           */
/* Readings:                                                                 */
/*  - defer: when delivery needs next_obs, the newest transition cannot be   */
/*    sampled yet (its successor does not exist).  Its leaf stays 0 and its  */
/*    priority waits in `pending` until the next insertion.                  */
/*  - q == NULL on insertion: PER's "new transitions get the maximal         */
/*    priority seen so far"; the running maximum starts at 1.0 (2^20) and   */
/*    covers every priority ever set.                                        */
/* ------------------------------------------------------------------------ */
ORC_API void orc_ingest_leaves(uint32_t *leaves, uint64_t cap, uint64_t total,
                               int defer, const uint32_t *q, uint64_t n,
                               uint32_t *pending, uint32_t *qmax) {
  for (uint64_t j = 0; j < n; ++j) {
    uint64_t id = total + j;
    uint32_t qj = q ? q[j] : *qmax;
    if (qj > *qmax) *qmax = qj;
    uint64_t slot = id % cap;
    if (defer) {
      if (id >= 1 && cap >= 2) leaves[(id - 1) % cap] = *pending;
      leaves[slot] = 0;
      *pending = qj;
    } else {
      leaves[slot] = qj;
    }
  }
}

/* Priority callback: pairs applied in batch order, so for a repeated index
 * the last occurrence wins.  A pair whose slot holds no transition, or whose
 * slot is >= cap, is skipped; the newest transition's priority goes to
 * `pending` when defer is set. */
ORC_API void orc_update_leaves(uint32_t *leaves, uint64_t cap, uint64_t total,
                               int defer, const int64_t *idx, const uint32_t *q,
                               uint64_t n, uint32_t *pending, uint32_t *qmax) {
  uint64_t size = orc_ring_size(cap, total);
  for (uint64_t p = 0; p < n; ++p) {
    if (idx[p] < 0 || (uint64_t)idx[p] >= cap) continue;
    uint64_t s = (uint64_t)idx[p];
    uint64_t k = orc_ring_offset(cap, total, s);
    if (k >= size) continue;
    if (q[p] > *qmax) *qmax = q[p];
    if (defer && k == size - 1)
      *pending = q[p];
    else
      leaves[s] = q[p];
  }
}

/* Sum of leaves[lo, hi), exact in 64 bits. */
ORC_API uint64_t orc_leaf_sum(const uint32_t *leaves, uint64_t lo, uint64_t hi) {
  uint64_t s = 0;
  for (uint64_t i = lo; i < hi; ++i) s += leaves[i];
  return s;
}

/* PER's proportional priority from a TD error: (|delta| + eps)^alpha, in
 * fp64, scaled by 2^20, rounded to nearest (ties to even), clamped to
 * [1, 2^32 - 1]. */
ORC_API uint32_t orc_priority_from_td(double td, double alpha, double eps) {
  double p = pow(fabs(td) + eps, alpha) * 1048576.0;
  double r = nearbyint(p);
  if (!(r >= 1.0)) r = 1.0;
  if (r > 4294967295.0) r = 4294967295.0;
  return (uint32_t)r;
}

ORC_API void orc_priorities_from_td(const float *td, uint64_t n, double alpha,
                                    double eps, uint32_t *q) {
  for (uint64_t i = 0; i < n; ++i) q[i] = orc_priority_from_td(td[i], alpha, eps);
}

/* ------------------------------------------------------------------------ */
/* Samplers (Sec. 2.2: off-policy delivery draws from the stored replay data). */
/* ------------------------------------------------------------------------ */

/* Uniform with replacement over the first n_valid logical offsets:
 * index_k = slot(mulhi64(u64(k; seed, round, stream 0), n_valid)). */
ORC_API void orc_sample_uniform(uint64_t cap, uint64_t total, uint64_t n_valid,
                                uint32_t B, uint64_t seed, uint64_t round,
                                int64_t *idx) {
  for (uint32_t k = 0; k < B; ++k) {
    uint64_t u = orc_philox_u64(seed, k, round, 0);
    uint64_t off = orc_mulhi64(u, n_valid);
    idx[k] = (int64_t)orc_ring_slot(cap, total, off);
  }
}

/* Stratified target of stratum k: [lo, hi) = [floor(kS/B), floor((k+1)S/B)),
 * t = lo + mulhi64(u, hi - lo), 128-bit intermediate products. */
ORC_API uint64_t orc_stratum_target(uint64_t S, uint32_t B, uint32_t k,
                                    uint64_t u) {
  unsigned __int128 lo = ((unsigned __int128)S * k) / B;
  unsigned __int128 hi = ((unsigned __int128)S * (k + 1)) / B;
  return (uint64_t)lo + orc_mulhi64(u, (uint64_t)(hi - lo));
}

/* Proportional prioritized sampling by the inverse CDF, found with a plain
 * linear scan over physical slot order: the answer for target t is the
 * unique i with prefix(i) <= t < prefix(i) + q_i.  Returns 0, or -1 when the
 * total priority is 0. */
ORC_API int orc_sample_prioritized_scan(const uint32_t *leaves, uint64_t cap,
                                        uint32_t B, uint64_t seed,
                                        uint64_t round, int64_t *idx,
                                        uint32_t *qout) {
  uint64_t S = orc_leaf_sum(leaves, 0, cap);
  if (S == 0) return -1;
  for (uint32_t k = 0; k < B; ++k) {
    uint64_t t = orc_stratum_target(S, B, k, orc_philox_u64(seed, k, round, 1));
    uint64_t prefix = 0;
    uint64_t i = 0;
    for (; i < cap; ++i) {
      if (t < prefix + leaves[i]) break;
      prefix += leaves[i];
    }
    idx[k] = (int64_t)i;
    qout[k] = leaves[i];
  }
  return 0;
}

/* The same inverse CDF through one exclusive-prefix array and a binary
 * search (largest i with prefix(i) <= t and q_i > 0). */
ORC_API int orc_sample_prioritized_bisect(const uint32_t *leaves, uint64_t cap,
                                          uint32_t B, uint64_t seed,
                                          uint64_t round, int64_t *idx,
                                          uint32_t *qout) {
  uint64_t *prefix = (uint64_t *)malloc((cap + 1) * sizeof(uint64_t));
  if (!prefix) return -2;
  prefix[0] = 0;
  for (uint64_t i = 0; i < cap; ++i) prefix[i + 1] = prefix[i] + leaves[i];
  uint64_t S = prefix[cap];
  if (S == 0) {
    free(prefix);
    return -1;
  }
  for (uint32_t k = 0; k < B; ++k) {
    uint64_t t = orc_stratum_target(S, B, k, orc_philox_u64(seed, k, round, 1));
    /* first i with prefix[i+1] > t */
    uint64_t lo = 0, hi = cap - 1;
    while (lo < hi) {
      uint64_t mid = lo + (hi - lo) / 2;
      if (prefix[mid + 1] > t)
        hi = mid;
      else
        lo = mid + 1;
    }
    idx[k] = (int64_t)lo;
    qout[k] = leaves[lo];
  }
  free(prefix);
  return 0;
}

/* Importance-sampling weights, PER: w_i = (N P(i))^-beta / max_j w_j with
 * the maximum taken over the batch; since P(i) = q_i / S this is
 * (q_min / q_i)^beta.  fp64, rounded once to fp32. */
ORC_API void orc_is_weights(const uint32_t *q, uint32_t B, double beta,
                            float *w) {
  uint32_t qmin = 0xFFFFFFFFu;
  for (uint32_t k = 0; k < B; ++k)
    if (q[k] < qmin) qmin = q[k];
  for (uint32_t k = 0; k < B; ++k)
    w[k] = (float)pow((double)qmin / (double)q[k], beta);
}

/* ------------------------------------------------------------------------ */
/* Byte -> float transforms used by delivery ("transform" step, Sec. 2.2).   */
/* ------------------------------------------------------------------------ */

/* x = fl32(b / 255): one correctly rounded IEEE binary32 division. */
ORC_API float orc_unit_f32(uint8_t b) {
  float num = (float)b;
  float den = 255.0f;
  return num / den;
}

/* Round a binary32 value to bfloat16, to nearest, ties to even. */
ORC_API uint16_t orc_bf16_rne(float x) {
  uint32_t u;
  memcpy(&u, &x, 4);
  if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) /* NaN */
    return (uint16_t)((u >> 16) | 0x40u);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

/* Per-channel normalisation: RNE_bf16(fl32(fl32(fl32(b/255) - mean) / std)),
 * every step rounded separately. */
ORC_API uint16_t orc_norm_bf16(uint8_t b, float mean, float stdv) {
  float x = orc_unit_f32(b);
  float t = x - mean;
  float y = t / stdv;
  return orc_bf16_rne(y);
}

/* ------------------------------------------------------------------------ */
/* Frame-stack delivery (Sec. 2.2: delivery materialises the chosen          */
/* transitions, concatenating and reshaping them; frame stacking of          */
/* Mnih et al., Nature 2015).  Readings:                                     */
/*  - obs(i) = [f(i-K+1), ..., f(i)] over logical predecessors; f(j) is an   */
/*    all-zero frame when j precedes the oldest stored transition or when    */
/*    any transition in [j, i-1] ended its episode (done == 1);              */
/*  - next_obs(i) = obs(i+1) by the same rule (so when done[i] == 1 it is    */
/*    [0, ..., 0, f(i+1)]);                                                  */
/*  - output values are fl32(byte/255).                                      */
/* One sample: anchor slot `slot`; frames [cap][F]; done [cap].             */
/* ------------------------------------------------------------------------ */
static void stack_at(const uint8_t *frames, const uint8_t *done, uint64_t cap,
                     uint64_t total, uint32_t F, uint32_t K, int64_t anchor_off,
                     float *out) {
  for (uint32_t m = 0; m < K; ++m) {
    int64_t j = anchor_off - (int64_t)(K - 1) + (int64_t)m;
    int zero = (j < 0);
    for (int64_t o = j; !zero && o < anchor_off; ++o)
      if (done[orc_ring_slot(cap, total, (uint64_t)o)]) zero = 1;
    float *dst = out + (uint64_t)m * F;
    if (zero) {
      for (uint32_t x = 0; x < F; ++x) dst[x] = 0.0f;
    } else {
      const uint8_t *src = frames + orc_ring_slot(cap, total, (uint64_t)j) * F;
      for (uint32_t x = 0; x < F; ++x) dst[x] = orc_unit_f32(src[x]);
    }
  }
}

ORC_API void orc_dqn_stack(const uint8_t *frames, const uint8_t *done,
                           uint64_t cap, uint64_t total, uint32_t F, uint32_t K,
                           int64_t slot, float *obs, float *next_obs) {
  int64_t k = (int64_t)orc_ring_offset(cap, total, (uint64_t)slot);
  stack_at(frames, done, cap, total, F, K, k, obs);
  if (next_obs) stack_at(frames, done, cap, total, F, K, k + 1, next_obs);
}

/* Batch form: obs/next_obs [B][K][F] float, plus collated action, reward,
 * done of the anchor transition. */
ORC_API void orc_deliver_dqn(const uint8_t *frames, const uint8_t *done,
                             const int32_t *action, const float *reward,
                             uint64_t cap, uint64_t total, uint32_t F,
                             uint32_t K, const int64_t *idx, uint32_t B,
                             float *obs, float *next_obs, int32_t *act_out,
                             float *rew_out, uint8_t *done_out) {
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < (int64_t)B; ++b) {
    int64_t s = idx[b];
    orc_dqn_stack(frames, done, cap, total, F, K, s,
                  obs + (uint64_t)b * K * F,
                  next_obs ? next_obs + (uint64_t)b * K * F : NULL);
    if (act_out) act_out[b] = action[s];
    if (rew_out) rew_out[b] = reward[s];
    if (done_out) done_out[b] = done[s];
  }
}

/* ------------------------------------------------------------------------ */
/* On-policy mini-batch delivery (Sec. 2.2: delivery partitions trajectories */
/* into mini-batches with shuffling).  Stored observation HWC uint8,         */
/* delivered CHW bfloat16 RNE(fl32(b/255)); per-sample scalars (advantage,   */
/* return) are gathered by the sample's logical offset.                      */
/* ------------------------------------------------------------------------ */
ORC_API void orc_hwc_to_chw_bf16(const uint8_t *hwc, uint32_t H, uint32_t W,
                                 uint32_t C, uint16_t *chw) {
  for (uint32_t c = 0; c < C; ++c)
    for (uint32_t y = 0; y < H; ++y)
      for (uint32_t x = 0; x < W; ++x)
        chw[((uint64_t)c * H + y) * W + x] =
            orc_bf16_rne(orc_unit_f32(hwc[((uint64_t)y * W + x) * C + c]));
}

ORC_API void orc_deliver_ppo(const uint8_t *obs_ring, uint64_t cap,
                             uint64_t total, uint32_t H, uint32_t W, uint32_t C,
                             const int64_t *idx, uint32_t B,
                             const float *adv_src, const float *ret_src,
                             uint16_t *obs_out, float *adv_out, float *ret_out) {
  uint64_t F = (uint64_t)H * W * C;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < (int64_t)B; ++b) {
    uint64_t s = (uint64_t)idx[b];
    orc_hwc_to_chw_bf16(obs_ring + s * F, H, W, C, obs_out + (uint64_t)b * F);
    uint64_t k = orc_ring_offset(cap, total, s);
    if (adv_out) adv_out[b] = adv_src[k];
    if (ret_out) ret_out[b] = ret_src[k];
  }
}

/* ------------------------------------------------------------------------ */
/* Multimodal delivery: stored CHW uint8 image, per-channel normalised       */
/* bfloat16, plus collated int32 tokens and reward.  The payload of one      */
/* sample is passed explicitly (so a caller can supply it from any tier).    */
/* ------------------------------------------------------------------------ */
ORC_API void orc_norm_chw_bf16(const uint8_t *chw, uint32_t C, uint64_t HW,
                               const float *mean, const float *stdv,
                               uint16_t *out) {
  for (uint32_t c = 0; c < C; ++c)
    for (uint64_t p = 0; p < HW; ++p)
      out[c * HW + p] = orc_norm_bf16(chw[c * HW + p], mean[c], stdv[c]);
}

ORC_API void orc_deliver_mm(const uint8_t *obs_ring, const int32_t *tok_ring,
                            const float *reward, uint32_t C, uint64_t HW,
                            uint32_t L, const int64_t *idx, uint32_t B,
                            const float *mean, const float *stdv,
                            uint16_t *obs_out, int32_t *tok_out,
                            float *rew_out) {
  uint64_t F = (uint64_t)C * HW;
#pragma omp parallel for schedule(static)
  for (int64_t b = 0; b < (int64_t)B; ++b) {
    uint64_t s = (uint64_t)idx[b];
    orc_norm_chw_bf16(obs_ring + s * F, C, HW, mean, stdv,
                      obs_out + (uint64_t)b * F);
    if (tok_out)
      memcpy(tok_out + (uint64_t)b * L, tok_ring + s * L, (size_t)L * 4);
    if (rew_out) rew_out[b] = reward[s];
  }
}

/* ------------------------------------------------------------------------ */
/* Generalized advantage estimation (Schulman et al., ICLR'16), the return  */
/* / advantage and normalisation steps of on-policy ingestion (Sec. 2.2).    */
/* Direct-sum definition, fp64:                                              */
/*   delta_t = r_t + gamma V_{t+1} (1 - d_t) - V_t                           */
/*   A_t = sum_{l >= 0, t+l < T} (gamma lambda)^l prod_{m<l}(1 - d_{t+m})    */
/*         delta_{t+l}                                                       */
/*   ret_t = A_t + V_t                                                       */
/* Layout: r, d [T][E]; v [T+1][E]; outputs [T][E].  Readings: d_t is the    */
/* done flag returned with r_t; V_T bootstraps the last step.                */
/* ------------------------------------------------------------------------ */
ORC_API void orc_gae(const float *r, const float *v, const uint8_t *d,
                     uint32_t T, uint32_t E, double gamma, double lambda,
                     double *adv, double *ret) {
#pragma omp parallel for schedule(static)
  for (int64_t e = 0; e < (int64_t)E; ++e) {
    for (uint32_t t = 0; t < T; ++t) {
      double A = 0.0;
      double coef = 1.0;
      for (uint32_t u = t; u < T; ++u) {
        uint64_t at = (uint64_t)u * E + e;
        double nd = d[at] ? 0.0 : 1.0;
        double delta = (double)r[at] +
                       gamma * (double)v[(uint64_t)(u + 1) * E + e] * nd -
                       (double)v[at];
        A += coef * delta;
        if (d[at]) break;
        coef *= gamma * lambda;
      }
      uint64_t o = (uint64_t)t * E + e;
      adv[o] = A;
      ret[o] = A + (double)v[o];
    }
  }
}

/* Global advantage normalisation: (A - mean) / (std + 1e-8), std with the
 * unbiased (n - 1) divisor, two passes in fp64. */
ORC_API void orc_normalize(const double *a, uint64_t n, double *out,
                           double *mean_out, double *std_out) {
  double s = 0.0;
  for (uint64_t i = 0; i < n; ++i) s += a[i];
  double mean = s / (double)n;
  double ss = 0.0;
  for (uint64_t i = 0; i < n; ++i) ss += (a[i] - mean) * (a[i] - mean);
  double sd = n > 1 ? sqrt(ss / (double)(n - 1)) : 0.0;
  for (uint64_t i = 0; i < n; ++i) out[i] = (a[i] - mean) / (sd + 1e-8);
  if (mean_out) *mean_out = mean;
  if (std_out) *std_out = sd;
}

/* ------------------------------------------------------------------------ */
/* Shuffle into mini-batches (Sec. 2.2 on-policy delivery; Appendix C        */
/* Invariant 2 requires the mini-batches of an iteration to partition its    */
/* rollout).  Reading: random-key sort, key_j = u64(j; seed, iteration,      */
/* stream 2), sorted ascending by (key, j).                                  */
/* ------------------------------------------------------------------------ */
typedef struct {
  uint64_t key;
  uint32_t j;
} orc_kj;

static int cmp_kj(const void *a, const void *b) {
  const orc_kj *x = (const orc_kj *)a, *y = (const orc_kj *)b;
  if (x->key != y->key) return x->key < y->key ? -1 : 1;
  if (x->j != y->j) return x->j < y->j ? -1 : 1;
  return 0;
}

ORC_API int orc_permutation(uint32_t n, uint64_t seed, uint64_t iteration,
                            int64_t *perm) {
  orc_kj *v = (orc_kj *)malloc((size_t)n * sizeof(orc_kj));
  if (!v) return -2;
  for (uint32_t j = 0; j < n; ++j) {
    v[j].key = orc_philox_u64(seed, j, iteration, 2);
    v[j].j = j;
  }
  qsort(v, n, sizeof(orc_kj), cmp_kj);
  for (uint32_t r = 0; r < n; ++r) perm[r] = v[r].j;
  free(v);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Two-tier placement (Sec. 5: the buffer is split across memory tiers --    */
/* pinned CPU and GPU among the candidate placements).  Reading: the newest  */
/* min(total, cap_h) transitions live in the HBM ring at slot L mod cap_h,   */
/* the older ones (down to the oldest retained) in the host ring at slot     */
/* L mod (cap - cap_h).  tier: 0 = HBM, 1 = host, -1 = not retained.         */
/* ------------------------------------------------------------------------ */
ORC_API void orc_tier_of(uint64_t cap, uint64_t cap_h, uint64_t total,
                         uint64_t L, int32_t *tier, uint64_t *slot) {
  uint64_t size = orc_ring_size(cap, total);
  uint64_t in_hbm = total < cap_h ? total : cap_h;
  if (L >= total || L < total - size) {
    *tier = -1;
    *slot = 0;
  } else if (L >= total - in_hbm) {
    *tier = 0;
    *slot = L % cap_h;
  } else {
    *tier = 1;
    *slot = L % (cap - cap_h);
  }
}
