// k_shard.cu -- the device side of a buffer sharded across G GPUs (the
// shared-GPU placement of Sec. 5.1: the ring's slots are split between the
// GPUs of a node and every learner samples the whole buffer, so most of a
// batch comes from other GPUs).
//
// The global prioritized distribution is the one of a single buffer whose
// leaves are the shards' leaves in shard-major order (shard 0's physical
// slots, then shard 1's, ...): its prefix sum up to shard s is
// P_s = S_0 + ... + S_{s-1}.  A round then needs one exchange:
//   1. every shard's total S_s (edp_tree_total), all-gathered;
//   2. each learner computes the stratified targets of its strata over
//      S = sum S_s -- the same targets a single buffer's sampler draws -- and
//      routes each to the shard whose prefix range [P_s, P_s + S_s) holds it,
//      as the local target t - P_s (k_route_prio); targets never decrease
//      with the stratum, so the routed list is grouped by shard, in stratum
//      order within each group;
//   3. the owners descend their own trees (k_sample_targets in k_tree.cu)
//      and deliver the rows, which travel back in the same grouping, so a
//      learner's rows arrive in stratum order;
//   4. importance weights take the minimum priority over the whole global
//      batch: each learner's minimum (k_batch_qmin), reduced over ranks, then
//      (q_min / q_k)^beta per row (k_is_weights).
// The collectives themselves run in the caller's communication library.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr uint32_t kMaxShards = 1024;
constexpr int kRouteThreads = 256;

__global__ void k_tree_total(const uint64_t *__restrict__ root, uint64_t *__restrict__ out) {
  pdl_wait();
  pdl_launch();
  if (threadIdx.x == 0) *out = *root;
}

// Strata [k0, k0 + n) of a batch of B over the shards' totals: local
// targets in stratum order and per-shard counts.  One CTA (a round routes a
// few hundred strata; the work is a Philox draw and a binary search each).
__global__ void __launch_bounds__(kRouteThreads)
k_route_prio(const uint64_t *__restrict__ totals, uint32_t G, uint32_t B, uint32_t k0,
             uint32_t n, uint64_t seed, uint64_t round, uint64_t *__restrict__ local_t,
             int64_t *__restrict__ counts, Ctrl *ctrl) {
  __shared__ uint64_t prefix[kMaxShards + 1];
  __shared__ uint32_t cnt[kMaxShards];
  __shared__ int bad;
  pdl_wait();
  pdl_launch();
  for (uint32_t s = threadIdx.x; s < G; s += kRouteThreads) cnt[s] = 0;
  if (threadIdx.x == 0) {
    // shard-major prefix sums; a total that does not fit in 64 bits is
    // reported and routes nothing
    uint64_t acc = 0;
    int overflow = 0;
    prefix[0] = 0;
    for (uint32_t s = 0; s < G; ++s) {
      const uint64_t v = totals[s];
      overflow |= acc + v < acc;
      acc += v;
      prefix[s + 1] = acc;
    }
    bad = overflow ? 2 : (acc == 0 ? 1 : 0);
    if (bad == 2) flag(ctrl, DEVERR_OVERFLOW, G);
    if (bad == 1 && n) flag(ctrl, DEVERR_EMPTY, k0);
  }
  __syncthreads();
  const uint64_t S = prefix[G];
  for (uint32_t i = threadIdx.x; i < n; i += kRouteThreads) {
    if (bad) {
      local_t[i] = ~0ull;  // no owner: an owner's descent reports it
      continue;
    }
    const uint64_t t = stratum_target(S, B, k0 + i, seed, round);
    // owner: the largest s < G with prefix[s] <= t (its total is then > 0)
    uint32_t lo = 0, hi = G;
    while (hi - lo > 1) {
      const uint32_t mid = (lo + hi) >> 1;
      if (prefix[mid] <= t) lo = mid; else hi = mid;
    }
    local_t[i] = t - prefix[lo];
    atomicAdd(&cnt[lo], 1u);
  }
  __syncthreads();
  for (uint32_t s = threadIdx.x; s < G; s += kRouteThreads) counts[s] = (int64_t)cnt[s];
}

// Minimum of q[0..n) as int64 (2^32 - 1 for n == 0, the neutral element of
// the minimum over ranks).  One CTA.
__global__ void __launch_bounds__(256)
k_batch_qmin(const uint32_t *__restrict__ q, uint32_t n, int64_t *__restrict__ out) {
  __shared__ uint32_t wmin[8];
  pdl_wait();
  pdl_launch();
  uint32_t m = 0xffffffffu;
  for (uint32_t i = threadIdx.x; i < n; i += 256) m = min(m, q[i]);
#pragma unroll
  for (int o = 16; o; o >>= 1) m = min(m, __shfl_xor_sync(0xffffffffu, m, o));
  if ((threadIdx.x & 31) == 0) wmin[threadIdx.x >> 5] = m;
  __syncthreads();
  if (threadIdx.x == 0) {
    for (int w = 1; w < 8; ++w) m = min(m, wmin[w]);
    *out = (int64_t)m;
  }
}

// w[k] = (q_min / q[k])^beta, fp64, one rounding to fp32 -- the delivery's
// importance weight with q_min given (the global batch minimum).
__global__ void k_is_weights(const uint32_t *__restrict__ q, uint32_t n,
                             const int64_t *__restrict__ qmin, double beta,
                             float *__restrict__ w) {
  pdl_wait();
  pdl_launch();
  const uint32_t m = (uint32_t)*qmin;
  for (uint32_t k = blockIdx.x * blockDim.x + threadIdx.x; k < n; k += gridDim.x * blockDim.x)
    w[k] = is_weight(m, q[k], beta);
}

}  // namespace

cudaError_t launch_tree_total(edp_ctx *c, uint64_t *total, cudaStream_t s) {
  return launch_pdl(k_tree_total, dim3(1), dim3(32), s, (const uint64_t *)c->level[0], total);
}

cudaError_t launch_route_prioritized(edp_ctx *c, const uint64_t *totals, uint32_t G,
                                     uint32_t B, uint32_t k0, uint32_t n, uint64_t seed,
                                     uint64_t round, uint64_t *local_t, int64_t *counts,
                                     cudaStream_t s) {
  if (G == 0 || G > kMaxShards) return cudaErrorInvalidValue;
  return launch_pdl(k_route_prio, dim3(1), dim3(kRouteThreads), s, totals, G, B, k0, n,
                    seed, round, local_t, counts, c->ctrl);
}

cudaError_t launch_batch_qmin(edp_ctx *c, const uint32_t *q, uint32_t n, int64_t *qmin,
                              cudaStream_t s) {
  (void)c;
  return launch_pdl(k_batch_qmin, dim3(1), dim3(256), s, q, n, qmin);
}

cudaError_t launch_is_weights(edp_ctx *c, const uint32_t *q, uint32_t n,
                              const int64_t *qmin, double beta, float *w, cudaStream_t s) {
  uint64_t blocks = (n + 255) / 256;
  if (blocks > 4ull * c->coop_sms) blocks = 4ull * c->coop_sms;
  if (blocks == 0) blocks = 1;
  return launch_pdl(k_is_weights, dim3((unsigned)blocks), dim3(256), s, q, n, qmin, beta, w);
}

}  // namespace edp
