// k_tree.cu -- the priority sum-tree of prioritized replay (Schaul et al.,
// ICLR'16; the replay-state callback of Appendix C, Invariant 2):
// refresh of ancestor sums, stratified inverse-CDF sampling by descent, and
// the priority update with last-occurrence-wins duplicate handling.
//
// Layout: a 32-ary tree in fixed point.  Leaves are the uint32 priorities of
// the ring slots (physical order, zero-padded to 32^D); level d < D holds
// 32^d uint64 sums, node n of level d covering leaves [n*32^(D-d),
// (n+1)*32^(D-d)).  Integer sums make every result independent of the order
// in which threads add, so sums, targets and indices are bit-exact.
//
// One warp serves one tree node: a level is one coalesced 256-byte (or
// 128-byte for leaves) load of the 32 children, a warp-shuffle inclusive
// prefix sum and a ballot -- D dependent loads per descent instead of the
// 5*D of a binary tree.
#include "edp_internal.cuh"

namespace edp {
namespace {

// Internal levels are stored back to back from the root: level d starts at
// node (32^d - 1) / 31.
struct TreeView {
  uint64_t *nodes;
  uint32_t *leaves;
  uint32_t depth;
  __device__ __forceinline__ uint64_t *lvl(uint32_t d) const {
    return nodes + (((1ull << (5 * d)) - 1) / 31);
  }
};

TreeView view(edp_ctx *c) {
  TreeView t{};
  t.nodes = c->level[0];
  t.leaves = c->leaves;
  t.depth = c->depth;
  return t;
}

constexpr unsigned kFull = 0xffffffffu;

__device__ __forceinline__ uint64_t warp_sum_u64(uint64_t v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// Recompute nodes [a0, a0+n0) and [a1, a1+n1) of level d from level d+1.
__global__ void k_tree_level(uint64_t *__restrict__ out,
                             const uint64_t *__restrict__ child64,
                             const uint32_t *__restrict__ child32, uint64_t a0,
                             uint64_t n0, uint64_t a1, uint64_t n1) {
  pdl_wait();
  pdl_launch();
  const uint64_t w = (blockIdx.x * (uint64_t)blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (w >= n0 + n1) return;
  const uint64_t node = w < n0 ? a0 + w : a1 + (w - n0);
  const uint64_t c = node * kFanout + lane;
  uint64_t v = child64 ? child64[c] : (uint64_t)child32[c];
  v = warp_sum_u64(v);
  if (lane == 0) out[node] = v;
}

// Stratified proportional sampling: one warp per stratum k.  The CTA first
// copies the top of the tree (levels 1 and 2: 32 + 1024 sums, 8.2 KiB) into
// shared memory, so a descent of a 1M-leaf tree makes two dependent global
// loads (level 3, then the leaf row) instead of four.
constexpr int kSmemLevels = 2;
constexpr int kSmemNodes = 32 + 1024;

// Copies levels 1 .. cached of the tree into top (all loads issued before
// any use); returns the number of cached levels.
__device__ __forceinline__ uint32_t cache_top(const TreeView &t, uint64_t *top,
                                              uint64_t keep) {
  const uint32_t cached = t.depth - 1 < (uint32_t)kSmemLevels ? t.depth - 1 : kSmemLevels;
  const uint32_t ncached = cached == 0 ? 0 : (cached == 1 ? 32 : 32 + 1024);
  uint64_t v5[5];
#pragma unroll
  for (int u = 0; u < 5; ++u) {
    const uint32_t i = threadIdx.x + u * 256;
    v5[u] = i < ncached ? ld_keep(t.nodes + 1 + i, keep) : 0ull;
  }
#pragma unroll
  for (int u = 0; u < 5; ++u) {
    const uint32_t i = threadIdx.x + u * 256;
    if (i < ncached) top[i] = v5[u];
  }
  return cached;
}

// Descent of one target (one warp): the leaf whose prefix range [prefix(i),
// prefix(i) + q_i) holds `target`, for target < S.  Per level: the 32
// children, an inclusive warp prefix sum and a ballot.  *ok is cleared if
// the sums disagree with the children (the leaf then stays in range).
__device__ __forceinline__ uint64_t descend(const TreeView &t, const uint64_t *top,
                                            uint32_t cached, uint64_t target, int lane,
                                            uint64_t keep, bool *ok) {
  uint64_t node = 0;
  for (uint32_t d = 1; d <= t.depth; ++d) {
    const uint64_t c = node * kFanout + lane;
    uint64_t v;
    if (d <= cached)
      v = top[(d == 1 ? 0 : 32) + c];
    else
      v = d < t.depth ? ld_keep(t.lvl(d) + c, keep) : (uint64_t)ld_keep(t.leaves + c, keep);
    uint64_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t y = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += y;
    }
    unsigned m = __ballot_sync(kFull, target < incl);
    if (m == 0) {  // sums disagree with children: report, stay in range
      *ok = false;
      m = 1u << 31;
    }
    const int f = __ffs(m) - 1;
    const uint64_t excl = __shfl_sync(kFull, incl - v, f);
    target = target >= excl ? target - excl : 0;
    node = node * kFanout + f;
  }
  return node;
}

__global__ void __launch_bounds__(256)
k_sample_prio(TreeView t, uint32_t B, uint64_t seed, uint64_t round,
              int64_t *__restrict__ idx, uint32_t *__restrict__ qout,
              Ctrl *ctrl) {
  __shared__ uint64_t top[kSmemNodes];
  const int lane = threadIdx.x & 31;
  const uint64_t keep = policy_keep();
  pdl_wait();
  const uint64_t S = t.nodes[0];  // issued beside the loads of the top levels
  const uint32_t cached = cache_top(t, top, keep);
  __syncthreads();
  const uint32_t warps = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t k = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; k < B;
       k += warps) {
    if (S == 0) {
      if (lane == 0) {
        idx[k] = -1;
        if (qout) qout[k] = 0;
        flag(ctrl, DEVERR_EMPTY, k);
      }
      continue;
    }
    const uint64_t target = stratum_target(S, B, k, seed, round);
    bool ok = true;
    const uint64_t node = descend(t, top, cached, target, lane, keep, &ok);
    if (lane == 0) {
      if (!ok) flag(ctrl, DEVERR_TREE, k);
      idx[k] = (int64_t)node;
      if (qout) qout[k] = t.leaves[node];
    }
  }
  pdl_launch();  // at the end: see pdl_launch()
}

// Descent of given targets (the shard side of a sharded buffer: targets
// routed here by edp_route_prioritized, each below this tree's total):
// one warp per target.  A target >= S is reported (DEVERR_INDEX) and
// gives idx -1, q 0.
__global__ void __launch_bounds__(256)
k_sample_targets(TreeView t, const uint64_t *__restrict__ targets, uint32_t n,
                 int64_t *__restrict__ idx, uint32_t *__restrict__ qout, Ctrl *ctrl) {
  __shared__ uint64_t top[kSmemNodes];
  const int lane = threadIdx.x & 31;
  const uint64_t keep = policy_keep();
  pdl_wait();
  const uint64_t S = t.nodes[0];  // issued beside the loads of the top levels
  const uint32_t cached = cache_top(t, top, keep);
  __syncthreads();
  const uint32_t warps = (gridDim.x * blockDim.x) >> 5;
  for (uint32_t k = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; k < n; k += warps) {
    const uint64_t target = targets[k];
    if (target >= S) {
      if (lane == 0) {
        idx[k] = -1;
        if (qout) qout[k] = 0;
        flag(ctrl, DEVERR_INDEX, target);
      }
      continue;
    }
    bool ok = true;
    const uint64_t node = descend(t, top, cached, target, lane, keep, &ok);
    if (lane == 0) {
      if (!ok) flag(ctrl, DEVERR_TREE, k);
      idx[k] = (int64_t)node;
      if (qout) qout[k] = t.leaves[node];
    }
  }
  pdl_launch();  // at the end: see pdl_launch()
}

// PER priority from a TD error: clamp(rn((|td| + eps)^alpha * 2^20), 1,
// 2^32 - 1) (the rule is defined in fp64).  The exponent, eps and the
// constants of the fast path travel as double-float splits made on the host.
struct PrioRule {
  double alpha, eps;
  float a_hi, a_lo, e_hi, e_lo;
  int fast;  // alpha in (0, 1], eps in [0, 2^90]: the double-float path applies
};

PrioRule prio_rule(double alpha, double eps) {
  PrioRule r{};
  r.alpha = alpha;
  r.eps = eps;
  r.a_hi = (float)alpha;
  r.a_lo = (float)(alpha - (double)r.a_hi);
  r.e_hi = (float)eps;
  r.e_lo = (float)(eps - (double)r.e_hi);
  r.fast = alpha > 0.0 && alpha <= 1.0 && eps >= 0.0 && eps <= 0x1p90;
  return r;
}

// x^a * 2^20 for x in [2^-100, 2^100] and a in (0, 1], rounded to the nearest
// integer and clamped, in double-float arithmetic.  An fp64 instruction
// occupies this GPU's fp64 pipe for about 64 cycles whatever the number of
// active lanes, so the fp64 evaluation of the rule costs ~4,000 cycles per
// warp; this one issues fp32 and integer work only.
//   log: x = 2^e m with m in [sqrt(1/2), sqrt(2)); ln m = 2 atanh(s),
//   s = (m - 1)/(m + 1), |s| <= 0.1716, by its series through s^17 (the
//   terms beyond s^7 in fp32: they are below 2^-17 relative to the sum);
//   exp: Cody and Waite's reduction t = n ln 2 + r, |r| <= ln(2)/2, with
//   ln 2 split into three floats (the first with 15 significant bits, so
//   that n times it is exact), and Taylor's series of e^r through r^12
//   (terms from r^7 on in fp32).
// Relative error below 2^-40: against the fp64 rule evaluated with the C
// library's pow, the integer differs in about one case per million, by one.
constexpr double kLn2 = 0.69314718055994530942;
constexpr float kLn2A = 0.693145751953125f;  // 0x3f317200
constexpr float kLn2B = (float)(kLn2 - (double)kLn2A);
constexpr float kLn2C = (float)(kLn2 - (double)kLn2A - (double)kLn2B);
#define EDP_DF_CONST(v) df{(float)(v), (float)((v) - (double)(float)(v))}

__device__ __forceinline__ df df_div(df a, df b) {
  const float q1 = __fdiv_rn(a.hi, b.hi);
  df r = df_add(a, df_mul_f(b, -q1));
  const float q2 = __fdiv_rn(r.hi, b.hi);
  r = df_add(r, df_mul_f(b, -q2));
  const float q3 = __fdiv_rn(r.hi, b.hi);
  return df_add_f(quick_two_sum(q1, q2), q3);
}

__device__ __forceinline__ df df_two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return {p, __fmaf_rn(a, b, -p)};
}

__device__ __forceinline__ uint32_t prio_df(df x, df a) {
  const int bits = __float_as_int(x.hi);
  int e = ((bits >> 23) & 0xff) - 127;
  if ((bits & 0x7fffff) > 0x3504f3) e += 1;  // mantissa above sqrt(2)
  const float sc = __int_as_float((127 - e) << 23);
  const df m{__fmul_rn(x.hi, sc), __fmul_rn(x.lo, sc)};
  const df s = df_div(df_add_f(m, -1.0f), df_add_f(m, 1.0f));
  const df s2 = df_mul(s, s);
  float tail = 1.0f / 17;
  tail = __fmaf_rn(tail, s2.hi, 1.0f / 15);
  tail = __fmaf_rn(tail, s2.hi, 1.0f / 13);
  tail = __fmaf_rn(tail, s2.hi, 1.0f / 11);
  tail = __fmaf_rn(tail, s2.hi, 1.0f / 9);
  df p = df_add(EDP_DF_CONST(1.0 / 7), df_mul_f(s2, tail));
  p = df_add(EDP_DF_CONST(1.0 / 5), df_mul(s2, p));
  p = df_add(EDP_DF_CONST(1.0 / 3), df_mul(s2, p));
  p = df_add_f(df_mul(s2, p), 1.0f);
  df lnm = df_mul(s, p);
  lnm.hi = __fmul_rn(lnm.hi, 2.0f);
  lnm.lo = __fmul_rn(lnm.lo, 2.0f);
  const float ef = (float)e;
  df el{__fmul_rn(ef, kLn2A), 0.0f};
  el = df_add(el, df_two_prod(ef, kLn2B));
  el = df_add_f(el, __fmul_rn(ef, kLn2C));
  const df t = df_mul(a, df_add(el, lnm));
  const float nf = rintf(__fmul_rn(t.hi, 1.44269504f));
  df r = df_add_f(t, -__fmul_rn(nf, kLn2A));
  r = df_add(r, df_two_prod(-nf, kLn2B));
  r = df_add_f(r, -__fmul_rn(nf, kLn2C));
  float qt = 1.0f / 479001600;
  qt = __fmaf_rn(qt, r.hi, 1.0f / 39916800);
  qt = __fmaf_rn(qt, r.hi, 1.0f / 3628800);
  qt = __fmaf_rn(qt, r.hi, 1.0f / 362880);
  qt = __fmaf_rn(qt, r.hi, 1.0f / 40320);
  qt = __fmaf_rn(qt, r.hi, 1.0f / 5040);
  df q = df_add(EDP_DF_CONST(1.0 / 720), df_mul_f(r, qt));
  q = df_add(EDP_DF_CONST(1.0 / 120), df_mul(r, q));
  q = df_add(EDP_DF_CONST(1.0 / 24), df_mul(r, q));
  q = df_add(EDP_DF_CONST(1.0 / 6), df_mul(r, q));
  q = df_add_f(df_mul(r, q), 0.5f);
  q = df_add_f(df_mul(r, q), 1.0f);
  q = df_add_f(df_mul(r, q), 1.0f);
  const float sc2 = __int_as_float((127 + (int)nf + 20) << 23);  // 2^(n + 20)
  const float vh = __fmul_rn(q.hi, sc2), vl = __fmul_rn(q.lo, sc2);
  if (vh >= 4294967296.0f) return 0xffffffffu;
  const float rh = rintf(vh);
  const float d = __fadd_rn(__fsub_rn(vh, rh), vl);
  long long res = (long long)rh + (long long)rintf(d);
  if (res < 1) res = 1;
  if (res > 4294967295ll) res = 4294967295ll;
  return (uint32_t)res;
}
#undef EDP_DF_CONST

__device__ __forceinline__ uint32_t prio_td(float td, const PrioRule &rule) {
  if (rule.fast) {
    const df x = df_add_f(df{rule.e_hi, rule.e_lo}, fabsf(td));
    if (x.hi >= 0x1p-100f && x.hi <= 0x1p100f) return prio_df(x, df{rule.a_hi, rule.a_lo});
  }
  // the fp64 evaluation: exponents outside (0, 1], and arguments far from 1
  const double x = fabs((double)td) + rule.eps;
  double p = (x > 1e-300 && x < 1e300) ? pow_pos<true>(x, rule.alpha) * 1048576.0
                                       : pow(x, rule.alpha) * 1048576.0;
  double r = rint(p);
  if (!(r >= 1.0)) r = 1.0;
  if (r > 4294967295.0) r = 4294967295.0;
  return (uint32_t)r;
}

__global__ void k_prio_from_td(const float *__restrict__ td, uint32_t n, PrioRule rule,
                               uint32_t *__restrict__ q) {
  for (uint32_t i = blockIdx.x * blockDim.x + threadIdx.x; i < n;
       i += gridDim.x * blockDim.x)
    q[i] = prio_td(td[i], rule);
}

constexpr int kUpdThreads = 512;
constexpr int kUpdPer = 2;                          // pairs per thread per chunk
constexpr int kUpdChunk = kUpdThreads * kUpdPer;
constexpr int kUpdTable = 2 * kUpdChunk;            // open-addressing table
constexpr uint32_t kEmpty = 0xffffffffu;

__device__ __forceinline__ uint32_t tab_hash(uint32_t x, uint32_t mask) {
  x ^= x >> 16;
  x *= 0x45d9f3bu;
  x ^= x >> 16;
  return x & mask;
}

// Priority update of a large batch (more than kUpdSmallMax pairs; smaller
// ones take k_update_small below).  Phase 1 (all CTAs): the priority of every pair -- the
// given u32, or PER's rule from the TD error, whose fp64 pow is spread over
// the CTAs -- goes to qbuf.  The last CTA to finish (ticket counter, no
// waiting) then applies the pairs in batch order, in chunks of 1024 (two
// pairs per thread): a shared-memory hash table keeps, per slot, the largest
// batch position (atomicMax), so only the last occurrence of a slot writes
// its leaf.  The
// exact signed delta of each written leaf is added to its ancestors
// (two's complement wrap makes negative deltas exact); the two top levels,
// which every pair shares, are summed on chip first.
__global__ void __launch_bounds__(kUpdThreads, 1)
k_update(TreeView t, const int64_t *__restrict__ idx,
         const uint32_t *__restrict__ q, const float *__restrict__ td,
         uint32_t *__restrict__ qbuf, PrioRule rule, uint32_t n,
         uint64_t cap, uint64_t oldest, uint64_t size, int defer, Ctrl *ctrl) {
  __shared__ uint32_t hkey[kUpdTable];
  __shared__ uint32_t hpos[kUpdTable];
  __shared__ uint32_t ticket;
  __shared__ uint32_t acc_lo[32], acc_hi[32];
  __shared__ unsigned long long warp_root[kUpdThreads / 32];
  const uint32_t *qv_src = q;
  // Nothing is read or written before the wait on the preceding kernel: it
  // may be the kernel that writes the TD errors, or the previous update,
  // whose last CTA may still be reading qbuf.
  pdl_wait();
  pdl_launch();
  if (td) {
    // phase 1: one warp per CTA, one CTA per 32 pairs, so the fp64 work
    // spreads over SMs
    if (threadIdx.x < 32)
      for (uint32_t p = blockIdx.x * 32 + threadIdx.x; p < n; p += gridDim.x * 32)
        qbuf[p] = prio_td(td[p], rule);
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) ticket = atomicAdd(&ctrl->upd_count, 1u);
    __syncthreads();
    if (ticket != gridDim.x - 1) return;
    __threadfence();
    qv_src = qbuf;
  } else if (blockIdx.x != 0) {
    return;
  }
  const uint32_t tsize = n >= kUpdChunk ? kUpdTable
                                        : max(64u, 2u << (31 - __clz(max(n, 1u))));
  const uint32_t mask = tsize - 1;
  uint32_t qmax_local = 0;  // running maximum: one atomic per CTA at the end
  const int lane = threadIdx.x & 31;
  unsigned long long root_sum = 0;
  if (threadIdx.x < 32) {
    acc_lo[threadIdx.x] = 0;
    acc_hi[threadIdx.x] = 0;
  }
  for (uint32_t base = 0; base < n; base += kUpdChunk) {
    const uint32_t cnt = min((uint32_t)kUpdChunk, n - base);
    for (uint32_t i = threadIdx.x; i < tsize; i += kUpdThreads) {
      hkey[i] = kEmpty;
      hpos[i] = 0;
    }
    __syncthreads();
    // every load of the chunk (index, priority, old leaf) is issued before
    // the barrier; pairs are read in batch order p = r * threads + tid
    int64_t s_[kUpdPer];
    uint32_t qv_[kUpdPer], old_[kUpdPer];
    uint64_t k_[kUpdPer];
    bool holds_[kUpdPer];
#pragma unroll
    for (int r = 0; r < kUpdPer; ++r) {
      const uint32_t p = r * kUpdThreads + threadIdx.x;
      const bool active = p < cnt;
      const int64_t sl = active ? idx[base + p] : -1;
      const bool valid = active && sl >= 0 && (uint64_t)sl < cap;
      if (active && !valid) flag(ctrl, DEVERR_INDEX, (unsigned long long)sl);
      const uint64_t k = !valid ? 0
                       : (uint64_t)sl >= oldest ? (uint64_t)sl - oldest
                                                : (uint64_t)sl + cap - oldest;
      const bool holds = valid && k < size;  // the slot holds a transition
      s_[r] = sl;
      k_[r] = k;
      holds_[r] = holds;
      qv_[r] = holds ? __ldcg(qv_src + base + p) : 0u;
      old_[r] = holds ? t.leaves[sl] : 0u;
      if (holds) {
        const uint32_t key = (uint32_t)sl;
        uint32_t h = tab_hash(key, mask);
        for (uint32_t probe = 0; probe < tsize; ++probe) {
          const uint32_t prev = atomicCAS(&hkey[h], kEmpty, key);
          if (prev == kEmpty || prev == key) {
            atomicMax(&hpos[h], p);
            break;
          }
          h = (h + 1) & mask;
        }
      }
    }
    __syncthreads();
#pragma unroll
    for (int r = 0; r < kUpdPer; ++r) {
      const uint32_t p = r * kUpdThreads + threadIdx.x;
      const int64_t sl = s_[r];
      const uint32_t qv = qv_[r];
      qmax_local = max(qmax_local, qv);
      bool win = false;
      if (holds_[r]) {
        uint32_t h = tab_hash((uint32_t)sl, mask);
        for (uint32_t probe = 0; probe < tsize && hkey[h] != (uint32_t)sl; ++probe)
          h = (h + 1) & mask;
        win = hpos[h] == p;  // no later pair sets this slot
      }
      if (win && defer && k_[r] == size - 1) {
        ctrl->pending_q = qv;
        win = false;
      }
      unsigned long long delta = 0;
      if (win) {
        t.leaves[sl] = qv;
        delta = (unsigned long long)((long long)qv - (long long)old_[r]);
      }
      // ancestors.  The root and level 1 (32 nodes) are shared by many
      // pairs: the root delta is summed over the block (shuffles, then one
      // atomic), level-1 deltas go to 32 shared accumulators kept as two
      // 32-bit halves with explicit carries (exact mod 2^64).  Deeper nodes
      // rarely collide and take one 64-bit atomic per pair.
      root_sum += delta;
      if (delta && t.depth >= 2) {
        const uint32_t n1 = (uint32_t)((uint64_t)sl >> (5 * (t.depth - 1)));
        const uint32_t lo = (uint32_t)delta, hi = (uint32_t)(delta >> 32);
        const uint32_t old = atomicAdd(&acc_lo[n1], lo);
        atomicAdd(&acc_hi[n1], hi + (old + lo < old ? 1u : 0u));
      }
      if (delta)
        for (uint32_t d = 2; d < t.depth; ++d)
          atomicAdd((unsigned long long *)&t.lvl(d)[(uint64_t)sl >> (5 * (t.depth - d))],
                    delta);
    }
    // flush the chunk's root and level-1 sums
#pragma unroll
    for (int o = 16; o; o >>= 1) root_sum += __shfl_xor_sync(kFull, root_sum, o);
    if (lane == 0) warp_root[threadIdx.x >> 5] = root_sum;
    root_sum = 0;
    __syncthreads();
    if (threadIdx.x < 32 && t.depth >= 2) {
      const unsigned long long v =
          ((unsigned long long)acc_hi[threadIdx.x] << 32) | acc_lo[threadIdx.x];
      if (v) atomicAdd((unsigned long long *)&t.lvl(1)[threadIdx.x], v);
      acc_lo[threadIdx.x] = 0;
      acc_hi[threadIdx.x] = 0;
    }
    if (threadIdx.x == 32) {
      unsigned long long v = 0;
      for (int w = 0; w < kUpdThreads / 32; ++w) v += warp_root[w];
      if (v) atomicAdd((unsigned long long *)&t.nodes[0], v);
    }
    __syncthreads();
  }
#pragma unroll
  for (int o = 16; o; o >>= 1)
    qmax_local = max(qmax_local, __shfl_xor_sync(kFull, qmax_local, o));
  if ((threadIdx.x & 31) == 0) ticket = 0;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) atomicMax(&ticket, qmax_local);
  __syncthreads();
  if (threadIdx.x == 0) {
    if (ticket) atomicMax(&ctrl->max_q, ticket);
    if (td) ctrl->upd_count = 0;  // ready for the next call
  }
}

// Priority update of a small batch (n <= kUpdSmallMax pairs): one CTA per 32
// pairs and a single pass, with no ticket and no second phase.  Each CTA
// stages the slots of the whole batch in shared memory and checks, for each
// of its own 32 pairs, whether a later pair of the batch sets the same slot
// (the table warps split the batch between them; every comparison reads one
// broadcast word).  The pairs that are the last occurrence of their slot
// write their leaves and add their exact deltas to the ancestors with
// atomics: each slot has exactly one writer in the batch, and integer sums
// do not depend on the order of the additions, so the tree equals the one
// the sequential application gives.  Warp 0 holds the CTA's pairs and
// evaluates their priorities meanwhile.
constexpr int kUpdSmallMax = 2048;
constexpr int kUpdSmallThreads = 256;
constexpr int kUpdScan = kUpdSmallThreads - 32;                        // scanning threads
constexpr int kUpdScanPer = (kUpdSmallMax + kUpdScan - 1) / kUpdScan;  // slots each loads

__global__ void __launch_bounds__(kUpdSmallThreads)
k_update_small(TreeView t, const int64_t *__restrict__ idx,
               const uint32_t *__restrict__ q, const float *__restrict__ td,
               PrioRule rule, uint32_t n, uint64_t cap, uint64_t oldest,
               uint64_t size, int defer, Ctrl *ctrl) {
  __shared__ uint32_t bkey[kUpdSmallMax];  // slot of each pair, kEmpty if it sets none
  __shared__ uint32_t later;               // bit l: a later pair sets pair l's slot
  __shared__ unsigned long long acc1[32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t p0 = blockIdx.x * 32, p = p0 + lane;  // warp 0's pair
  pdl_wait();
  pdl_launch();
  int64_t sl = -1;
  uint64_t k = 0;
  bool holds = false;
  uint32_t qv = 0, old = 0;
  if (warp == 0) {
    float tdv = 0.f;
    if (p < n) {
      sl = idx[p];
      if (td) tdv = td[p];
      else qv = q[p];
      const bool valid = sl >= 0 && (uint64_t)sl < cap;
      if (!valid) flag(ctrl, DEVERR_INDEX, (unsigned long long)sl);
      k = !valid ? 0
          : (uint64_t)sl >= oldest ? (uint64_t)sl - oldest : (uint64_t)sl + cap - oldest;
      holds = valid && k < size;  // the slot holds a transition
      if (holds) old = t.leaves[sl];
    }
    if (holds && td) qv = prio_td(tdv, rule);
    if (!holds) qv = 0;
  } else {
    // the slots of the whole batch, every load in flight at once
    const uint32_t f = threadIdx.x - 32;
#pragma unroll
    for (int j = 0; j < kUpdScanPer; ++j) {
      const uint32_t i = f + j * kUpdScan;
      if (i < n) {
        const int64_t s2 = idx[i];
        uint32_t key = kEmpty;
        if (s2 >= 0 && (uint64_t)s2 < cap) {
          const uint64_t k2 = (uint64_t)s2 >= oldest ? (uint64_t)s2 - oldest
                                                     : (uint64_t)s2 + cap - oldest;
          if (k2 < size) key = (uint32_t)s2;
        }
        bkey[i] = key;
      }
    }
    if (f == 0) later = 0;
    asm volatile("bar.sync 1, %0;" :: "r"(kUpdScan) : "memory");
    // scanning warp w - 1 compares the CTA's pairs (one per lane) with the
    // later pairs among [j0, j1); every lane reads the same word (a
    // broadcast), and the loop is the same for all lanes
    const uint32_t mine = p < n ? bkey[p] : kEmpty;
    const uint32_t per = (n + (kUpdScan / 32) - 1) / (kUpdScan / 32);
    const uint32_t j0 = (warp - 1) * per;
    const uint32_t j1 = min(n, j0 + per);
    uint32_t j = max(j0, p0 + 1);
    bool dup = false;
    for (; j + 8 <= j1; j += 8) {
#pragma unroll
      for (int u = 0; u < 8; ++u) dup |= (bkey[j + u] == mine) & (j + u > p);
    }
    for (; j < j1; ++j) dup |= (bkey[j] == mine) & (j > p);
    const unsigned m = __ballot_sync(kFull, dup && mine != kEmpty);
    if (lane == 0 && m) atomicOr(&later, m);
  }
  __syncthreads();
  if (warp != 0) return;
  bool win = holds && !((later >> lane) & 1u);  // no later pair sets this slot
  if (win && defer && k == size - 1) {
    ctrl->pending_q = qv;
    win = false;
  }
  unsigned long long delta = 0;
  if (win) {
    t.leaves[sl] = qv;
    delta = (unsigned long long)((long long)qv - (long long)old);
  }
  if (delta) {
    uint64_t first = 33;  // level d starts at node (32^d - 1) / 31
    for (uint32_t d = 2; d < t.depth; ++d, first = first * 32 + 1)
      atomicAdd((unsigned long long *)&t.nodes[first + ((uint64_t)sl >> (5 * (t.depth - d)))],
                delta);
  }
  if (t.depth >= 2) {  // level 1 (32 nodes): the warp's deltas per node first
    acc1[lane] = 0;
    __syncwarp();
    if (delta) atomicAdd(&acc1[(uint64_t)sl >> (5 * (t.depth - 1))], delta);
    __syncwarp();
    if (acc1[lane]) atomicAdd((unsigned long long *)&t.nodes[1 + lane], acc1[lane]);
  }
  const unsigned long long root = warp_sum_u64(delta);
  uint32_t qmax = qv;  // 0 for a pair that sets no leaf
#pragma unroll
  for (int o = 16; o; o >>= 1) qmax = max(qmax, __shfl_xor_sync(kFull, qmax, o));
  if (lane == 0) {
    if (root) atomicAdd((unsigned long long *)&t.nodes[0], root);
    if (qmax) atomicMax(&ctrl->max_q, qmax);
  }
}

}  // namespace

void tree_ranges(const edp_ctx *c, uint64_t first, uint64_t count, TreeRanges *out) {
  // leaf ranges [a0, b0) and [a1, b1) (the second only on ring wrap)
  uint64_t a0 = first, b0 = first + count, a1 = 0, b1 = 0;
  if (b0 > c->cap) {
    b1 = b0 - c->cap;
    b0 = c->cap;
  }
  for (int d = (int)c->depth - 1; d >= 0; --d) {
    const unsigned shift = 5u * (c->depth - d);
    uint64_t x0 = a0 >> shift, y0 = ((b0 - 1) >> shift) + 1;
    uint64_t x1 = 0, y1 = 0;
    if (b1 > a1) {
      x1 = a1 >> shift;
      y1 = ((b1 - 1) >> shift) + 1;
      if (y1 >= x0) {  // ranges meet: one range covers both
        x0 = x1 < x0 ? x1 : x0;
        y0 = y1 > y0 ? y1 : y0;
        x1 = y1 = 0;
      }
    }
    out->a0[d] = x0;
    out->n0[d] = y0 - x0;
    out->a1[d] = x1;
    out->n1[d] = y1 - x1;
  }
}

cudaError_t launch_tree_refresh(edp_ctx *c, uint64_t first, uint64_t count,
                                cudaStream_t s) {
  if (!c->depth || !count) return cudaSuccess;
  TreeRanges r;
  tree_ranges(c, first, count, &r);
  for (int d = (int)c->depth - 1; d >= 0; --d) {
    const uint64_t nodes = r.n0[d] + r.n1[d];
    const uint64_t threads = nodes * 32;
    const unsigned blocks = (unsigned)((threads + 255) / 256);
    const bool leaves_below = (uint32_t)(d + 1) == c->depth;
    cudaError_t e = launch_pdl(k_tree_level, dim3(blocks), dim3(256), s, c->level[d],
                               leaves_below ? (const uint64_t *)nullptr
                                            : (const uint64_t *)c->level[d + 1],
                               leaves_below ? (const uint32_t *)c->leaves
                                            : (const uint32_t *)nullptr,
                               r.a0[d], r.n0[d], r.a1[d], r.n1[d]);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_tree_build_all(edp_ctx *c, cudaStream_t s) {
  return launch_tree_refresh(c, 0, c->cap, s);
}

cudaError_t launch_sample_targets(edp_ctx *c, const uint64_t *targets, uint32_t n,
                                  int64_t *idx, uint32_t *q, cudaStream_t s) {
  const unsigned warps_per_block = 8;
  uint64_t blocks = (n + warps_per_block - 1) / warps_per_block;
  if (blocks > 8u * (unsigned)c->coop_sms) blocks = 8u * (unsigned)c->coop_sms;
  return launch_pdl(k_sample_targets, dim3((unsigned)blocks), dim3(warps_per_block * 32),
                    s, view(c), targets, n, idx, q, c->ctrl);
}

cudaError_t launch_sample_prioritized(edp_ctx *c, uint32_t B, uint64_t seed,
                                      uint64_t round, int64_t *idx, uint32_t *q,
                                      cudaStream_t s) {
  const unsigned warps_per_block = 8;
  uint64_t blocks = (B + warps_per_block - 1) / warps_per_block;
  if (blocks > 8u * (unsigned)c->coop_sms) blocks = 8u * (unsigned)c->coop_sms;
  return launch_pdl(k_sample_prio, dim3((unsigned)blocks), dim3(warps_per_block * 32),
                    s, view(c), B, seed, round, idx, q, c->ctrl);
}

cudaError_t launch_update(edp_ctx *c, const int64_t *idx, const uint32_t *q,
                          const float *td, double alpha, double eps, uint32_t n,
                          cudaStream_t s) {
  const uint64_t size = c->total < c->cap ? c->total : c->cap;
  const uint64_t oldest = (c->total - size) % c->cap;
  if (n <= (uint32_t)kUpdSmallMax)
    return launch_pdl(k_update_small, dim3((n + 31) / 32), dim3(kUpdSmallThreads), s,
                      view(c), idx, q, td, prio_rule(alpha, eps), n, c->cap, oldest,
                      size, c->defer, c->ctrl);
  uint32_t *qbuf = nullptr;
  unsigned grid = 1;
  if (td) {
    const cudaError_t e = ctx_qbuf(c, n, s, &qbuf);
    if (e != cudaSuccess) return e;
    // 32 priorities (one warp) per CTA: the fp64 work spreads over SMs
    grid = (n + 31) / 32;
    if (grid > 2u * (unsigned)c->coop_sms) grid = 2u * (unsigned)c->coop_sms;
  }
  return launch_pdl(k_update, dim3(grid), dim3(kUpdThreads), s, view(c), idx, q,
                    td, qbuf, prio_rule(alpha, eps), n, c->cap, oldest, size, c->defer,
                    c->ctrl);
}

cudaError_t launch_prio_from_td(const float *td, uint32_t n, double alpha,
                                double eps, uint32_t *q, cudaStream_t s) {
  const unsigned blocks = (n + 255) / 256 < 1024 ? (n + 255) / 256 : 1024;
  k_prio_from_td<<<blocks, 256, 0, s>>>(td, n, prio_rule(alpha, eps), q);
  return cudaGetLastError();
}

}  // namespace edp

// ---------------------------------------------------------------------------
// Allocation-free priority update.  Same kernels as edp_update_priorities_td:
// up to 2,048 pairs the single-pass kernel, which needs no memory beyond
// its arguments; above that the two-phase kernel, whose per-pair priorities
// computed from the TD errors go to the fixed array below instead of
// context-owned scratch that is allocated on first use.  Callers that must not allocate device memory use it: code being
// captured into a CUDA graph (cudaMalloc may not be called during stream
// capture), and runtimes that hand out all device memory up front and forbid
// allocation later, or that cannot afford the device-wide synchronisation a
// cudaMalloc/cudaFree may bring.  The array is per device and lives until
// the process exits; every call on that device shares it.  Calls queued on
// one stream are ordered (the kernel touches the array only after its wait
// on the preceding kernel); calls that can run at the same time on different
// streams race.  Nothing in it needs to start at zero: a call writes
// priorities [0, n) before it reads them.
// ---------------------------------------------------------------------------
#include <mutex>

namespace edp {
namespace {

constexpr uint32_t kStaticMaxPairs = 16384;  // 64 KiB of priorities
static __device__ __align__(256) uint32_t g_static_qbuf[kStaticMaxPairs];

constexpr int kMaxDevices = 64;
std::mutex g_static_mu;
uint32_t *g_static_ptr[kMaxDevices] = {};

// Device address of g_static_qbuf on the current device (looked up once per
// device; the host-side name is only a stand-in for the device symbol).
cudaError_t static_qbuf(int dev, uint32_t **out) {
  std::lock_guard<std::mutex> lock(g_static_mu);
  if (!g_static_ptr[dev]) {
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_static_qbuf);
    if (e != cudaSuccess) return e;
    g_static_ptr[dev] = (uint32_t *)p;
  }
  *out = g_static_ptr[dev];
  return cudaSuccess;
}

}  // namespace
}  // namespace edp

extern "C" edp_status edp_update_priorities_td_static(
    edp_ctx *ctx, const int64_t *idx, const float *td, uint32_t n,
    double alpha, double eps, edp_stream stream) {
  using namespace edp;
  static const char who[] = "edp_update_priorities_td_static";
  if (ctx && n && !td) return fail(ctx, EDP_ERR_INVALID, "%s: td NULL", who);
  const edp_status st = update_args(ctx, who, idx, nullptr, td, n, alpha, eps);
  if (st != EDP_OK || n == 0) return st;
  if (n > kStaticMaxPairs)
    return fail(ctx, EDP_ERR_INVALID,
                "%s: n exceeds the fixed maximum of 16384 pairs (use "
                "edp_update_priorities_td)", who);
  if (ctx->cfg.device < 0 || ctx->cfg.device >= kMaxDevices)
    return fail(ctx, EDP_ERR_INVALID, "%s: device ordinal out of range", who);
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(who);
  const uint64_t size = ctx->total < ctx->cap ? ctx->total : ctx->cap;
  const uint64_t oldest = (ctx->total - size) % ctx->cap;
  cudaError_t e;
  if (n <= (uint32_t)kUpdSmallMax) {  // needs no priority array
    e = launch_pdl(k_update_small, dim3((n + 31) / 32), dim3(kUpdSmallThreads),
                   (cudaStream_t)stream, view(ctx), idx, (const uint32_t *)nullptr, td,
                   prio_rule(alpha, eps), n, ctx->cap, oldest, size, ctx->defer, ctx->ctrl);
    if (e != cudaSuccess) {
      cudaGetLastError();
      return fail(ctx, EDP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
    }
    return EDP_OK;
  }
  uint32_t *qbuf = nullptr;
  e = static_qbuf(ctx->cfg.device, &qbuf);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(ctx, EDP_ERR_CUDA, "%s: cudaGetSymbolAddress: %s", who,
                cudaGetErrorString(e));
  }
  unsigned grid = (n + 31) / 32;
  if (grid > 2u * (unsigned)ctx->coop_sms) grid = 2u * (unsigned)ctx->coop_sms;
  e = launch_pdl(k_update, dim3(grid), dim3(kUpdThreads), (cudaStream_t)stream,
                 view(ctx), idx, (const uint32_t *)nullptr, td, qbuf, prio_rule(alpha, eps),
                 n, ctx->cap, oldest, size, ctx->defer, ctx->ctrl);
  if (e != cudaSuccess) {
    cudaGetLastError();
    return fail(ctx, EDP_ERR_CUDA, "%s: %s", who, cudaGetErrorString(e));
  }
  return EDP_OK;
}
