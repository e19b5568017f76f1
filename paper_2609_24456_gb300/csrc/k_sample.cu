// k_sample.cu -- the uniform replay sampler and the on-policy shuffle.
//
// Uniform: index_k = slot(mulhi64(Philox(k; seed, round, stream 0), n_valid)),
// one thread per index, no shared state.
//
// Shuffle (mini-batch partition with shuffling, Sec. 2.2 on-policy
// delivery): a random-key sort of the logical offsets j < n by
// (Philox(j; seed, round, stream 2), j), as three kernels chained with
// programmatic dependent launch (no grid-wide barrier):
//   keys     draw key_j, count it into bucket key_j >> (64 - log2 nb)
//   scatter  every CTA scans the nb <= 8192 counts in shared memory (the
//            bucket starts), then places its (key, j) pairs into their
//            buckets' ranges
//   rank     rank_j = bucket start + #{members < (key_j, j)}; idx[rank_j] =
//            slot of offset j; re-zero the counters for the next call
// With nb ~ n/4 buckets a bucket holds ~4 keys, so the in-bucket ranking is
// a handful of compares; the result does not depend on the scatter order.
#include "edp_internal.cuh"

namespace edp {
namespace {

__global__ void k_sample_uniform(uint32_t B, uint64_t seed, uint64_t round,
                                 uint64_t n_valid, uint64_t oldest,
                                 uint64_t cap, int64_t *__restrict__ idx) {
  pdl_wait();
  for (uint32_t k = blockIdx.x * blockDim.x + threadIdx.x; k < B;
       k += gridDim.x * blockDim.x) {
    const uint64_t off = mulhi64(philox_u64(seed, k, round, 0), n_valid);
    idx[k] = (int64_t)((oldest + off) % cap);
  }
  pdl_launch();  // at the end: see pdl_launch()
}

constexpr int kPermThreads = 256;
constexpr uint32_t kMaxBuckets = 8192;  // bucket starts scanned in shared memory

}  // namespace

size_t perm_scratch_bytes(uint32_t n) {
  return 3 * (kMaxBuckets + 64) * sizeof(uint32_t) + (size_t)n * (8 + 8 + 4 + 8) + 256;
}
size_t perm_zeroed_bytes() { return 2 * kMaxBuckets * sizeof(uint32_t); }

namespace {

struct PermScratch {
  uint32_t *count;   // [nb], zero between calls
  uint32_t *cursor;  // [nb], zero between calls
  uint32_t *start;   // [nb + 1] bucket starts
  uint64_t *keys;    // [n]
  uint64_t *lkey;    // [n] bucketed keys
  uint32_t *lj;      // [n] bucketed offsets
  uint2 *bounds;     // [n] each element's bucket [start, end)
};

__device__ __forceinline__ uint32_t bucket_of(uint64_t key, int lg) {
  return lg ? (uint32_t)(key >> (64 - lg)) : 0u;
}

__global__ void __launch_bounds__(kPermThreads)
k_perm_keys(uint32_t n, uint64_t seed, uint64_t round, int lg, PermScratch sc) {
  pdl_wait();
  pdl_launch();
  for (uint32_t j = blockIdx.x * kPermThreads + threadIdx.x; j < n;
       j += gridDim.x * kPermThreads) {
    const uint64_t key = philox_u64(seed, j, round, 2);
    sc.keys[j] = key;
    atomicAdd(&sc.count[bucket_of(key, lg)], 1u);
  }
}

// Exclusive scan of the nb bucket counts into smem start[] (padded layout:
// each thread scans 32 consecutive entries without bank conflicts).
__device__ __forceinline__ uint32_t pad32(uint32_t i) { return i + i / 32; }

__global__ void __launch_bounds__(kPermThreads)
k_perm_scatter(uint32_t n, int lg, PermScratch sc) {
  __shared__ uint32_t start[kMaxBuckets + kMaxBuckets / 32];
  __shared__ uint32_t warp_tot[kPermThreads / 32];
  const uint32_t nb = 1u << lg;
  pdl_wait();
  pdl_launch();
  for (uint32_t i = threadIdx.x; i < kMaxBuckets; i += kPermThreads)
    start[pad32(i)] = i < nb ? __ldcg(&sc.count[i]) : 0u;
  __syncthreads();
  constexpr uint32_t per = kMaxBuckets / kPermThreads;  // 32
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const uint32_t b0 = threadIdx.x * per;
  uint32_t run = 0;
#pragma unroll
  for (uint32_t i = 0; i < per; ++i) run += start[pad32(b0 + i)];
  uint32_t incl = run;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (lane >= o) incl += y;
  }
  if (lane == 31) warp_tot[wid] = incl;
  __syncthreads();
  uint32_t acc = incl - run;
  for (int w = 0; w < wid; ++w) acc += warp_tot[w];
#pragma unroll
  for (uint32_t i = 0; i < per; ++i) {
    const uint32_t k = pad32(b0 + i);
    const uint32_t cnt = start[k];
    start[k] = acc;
    acc += cnt;
  }
  __syncthreads();
  if (blockIdx.x == 0) {
    for (uint32_t i = threadIdx.x; i < nb; i += kPermThreads) sc.start[i] = start[pad32(i)];
    if (threadIdx.x == 0) sc.start[nb] = n;
  }
  for (uint32_t j = blockIdx.x * kPermThreads + threadIdx.x; j < n;
       j += gridDim.x * kPermThreads) {
    const uint64_t key = __ldcg(&sc.keys[j]);
    const uint32_t b = bucket_of(key, lg);
    const uint32_t lo = start[pad32(b)];
    const uint32_t pos = lo + atomicAdd(&sc.cursor[b], 1u);
    sc.lkey[pos] = key;
    sc.lj[pos] = j;
    sc.bounds[j] = make_uint2(lo, b + 1 < nb ? start[pad32(b + 1)] : n);
  }
}

__global__ void __launch_bounds__(kPermThreads)
k_perm_rank(uint32_t n, int lg, PermScratch sc, uint64_t oldest, uint64_t cap,
            int64_t *__restrict__ idx) {
  const uint32_t nb = 1u << lg;
  const uint32_t stride = gridDim.x * kPermThreads;
  const uint32_t tid = blockIdx.x * kPermThreads + threadIdx.x;
  pdl_wait();
  pdl_launch();
  for (uint32_t j = tid; j < n; j += stride) {
    const uint64_t key = __ldcg(&sc.keys[j]);
    const uint2 bd = __ldcg(&sc.bounds[j]);
    const uint32_t lo = bd.x, hi = bd.y;
    uint32_t r = 0;
    for (uint32_t i0 = lo; i0 < hi; i0 += 4) {  // members, 4 loads at a time
      uint64_t k2[4];
      uint32_t j2[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const bool in = i0 + u < hi;
        k2[u] = in ? __ldcg(&sc.lkey[i0 + u]) : ~0ull;
        j2[u] = in ? __ldcg(&sc.lj[i0 + u]) : 0xffffffffu;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) r += (k2[u] < key) || (k2[u] == key && j2[u] < j);
    }
    const uint64_t s2 = oldest + j;  // < 2 cap
    idx[lo + r] = (int64_t)(s2 >= cap ? s2 - cap : s2);
  }
  // this kernel reads only the bucket starts: the counters can be cleared
  // for the next call
  for (uint32_t b = tid; b < nb; b += stride) {
    sc.count[b] = 0;
    sc.cursor[b] = 0;
  }
}

}  // namespace

cudaError_t launch_sample_uniform(edp_ctx *c, uint32_t B, uint64_t seed,
                                  uint64_t round, int64_t *idx, cudaStream_t s) {
  const uint64_t size = c->total < c->cap ? c->total : c->cap;
  const uint64_t oldest = (c->total - size) % c->cap;
  const uint64_t nv = size - c->defer;
  const unsigned threads = 128;
  unsigned blocks = (B + threads - 1) / threads;
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(k_sample_uniform, dim3(blocks), dim3(threads), s, B, seed,
                    round, nv, oldest, c->cap, idx);
}

cudaError_t launch_permute(edp_ctx *c, uint32_t n, uint64_t seed,
                           uint64_t round, int64_t *idx, cudaStream_t s) {
  int lg = 0;
  while ((1ull << (lg + 2)) < n && (1u << lg) < kMaxBuckets) ++lg;  // nb ~ n/4
  const uint32_t nb = 1u << lg;
  void *block = nullptr;
  const cudaError_t ge = ctx_perm_scratch(c, perm_scratch_bytes(n), s, &block);
  if (ge != cudaSuccess) return ge;
  uint8_t *base = (uint8_t *)block;
  PermScratch sc;
  sc.count = (uint32_t *)base;  // the zeroed head of the block
  sc.cursor = sc.count + kMaxBuckets;
  sc.start = sc.cursor + kMaxBuckets;
  sc.keys = (uint64_t *)(base + 3 * (kMaxBuckets + 64) * sizeof(uint32_t));
  sc.lkey = sc.keys + n;
  sc.lj = (uint32_t *)(sc.lkey + n);
  sc.bounds = (uint2 *)(sc.lj + n + (n & 1));  // 8-byte aligned
  const uint64_t size = c->total < c->cap ? c->total : c->cap;
  const uint64_t oldest = (c->total - size) % c->cap;
  uint64_t grid = (n + kPermThreads - 1) / kPermThreads;
  if (grid > 4ull * c->coop_sms) grid = 4ull * c->coop_sms;
  const dim3 g((unsigned)grid), blk(kPermThreads);
  cudaError_t e = launch_pdl(k_perm_keys, g, blk, s, n, seed, round, lg, sc);
  if (e == cudaSuccess) e = launch_pdl(k_perm_scatter, g, blk, s, n, lg, sc);
  if (e == cudaSuccess)
    e = launch_pdl(k_perm_rank, g, blk, s, n, lg, sc, oldest, c->cap, idx);
  (void)nb;
  return e;
}

}  // namespace edp
