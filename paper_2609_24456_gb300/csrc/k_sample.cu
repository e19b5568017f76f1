// k_sample.cu -- the uniform replay sampler and the on-policy shuffle.
//
// Uniform: index_k = slot(mulhi64(Philox(k; seed, round, stream 0), n_valid)),
// one thread per index, no shared state.
//
// Shuffle (mini-batch partition with shuffling, Sec. 2.2 on-policy
// delivery): a random-key sort of the logical offsets j < n by
// (Philox(j; seed, round, stream 2), j).  One cooperative kernel:
//   phase 0  zero the bucket counters
//   phase 1  draw key_j, count it into bucket key_j >> (64 - log2 nb)
//   phase 2  exclusive scan of the counts (block 0)
//   phase 3  scatter (key, j) into its bucket's range
//   phase 4  rank_j = bucket start + #{members < (key_j, j)}; idx[rank_j] =
//            slot of offset j
// With nb ~ n/4 buckets a bucket holds ~4 keys, so the in-bucket ranking is
// a handful of compares; the result does not depend on the scatter order.
#include "edp_internal.cuh"

namespace edp {
namespace {

__global__ void k_sample_uniform(uint32_t B, uint64_t seed, uint64_t round,
                                 uint64_t n_valid, uint64_t oldest,
                                 uint64_t cap, int64_t *__restrict__ idx) {
  pdl_wait();
  pdl_launch();
  for (uint32_t k = blockIdx.x * blockDim.x + threadIdx.x; k < B;
       k += gridDim.x * blockDim.x) {
    const uint64_t off = mulhi64(philox_u64(seed, k, round, 0), n_valid);
    idx[k] = (int64_t)((oldest + off) % cap);
  }
}

constexpr int kPermThreads = 256;

struct PermScratch {
  uint32_t *count;    // [nb]
  uint32_t *cursor;   // [nb]
  uint32_t *offset;   // [nb + 1]
  uint64_t *keys;     // [n]
  uint64_t *lkey;     // [n] bucketed keys
  uint32_t *lj;       // [n] bucketed offsets
};

__device__ __forceinline__ uint32_t bucket_of(uint64_t key, int lg) {
  return lg ? (uint32_t)(key >> (64 - lg)) : 0u;
}

__global__ void __launch_bounds__(kPermThreads)
k_permute(uint32_t n, uint64_t seed, uint64_t round, int lg, PermScratch sc,
          uint64_t oldest, uint64_t cap, int64_t *__restrict__ idx, Ctrl *ctrl) {
  const uint32_t nb = 1u << lg;
  const uint32_t tid = blockIdx.x * kPermThreads + threadIdx.x;
  const uint32_t stride = gridDim.x * kPermThreads;
  // phase 0
  for (uint32_t b = tid; b < nb; b += stride) {
    sc.count[b] = 0;
    sc.cursor[b] = 0;
  }
  grid_barrier(ctrl, gridDim.x);
  // phase 1
  for (uint32_t j = tid; j < n; j += stride) {
    const uint64_t key = philox_u64(seed, j, round, 2);
    sc.keys[j] = key;
    atomicAdd(&sc.count[bucket_of(key, lg)], 1u);
  }
  grid_barrier(ctrl, gridDim.x);
  // phase 2: block 0 scans nb counts, per-thread runs + warp-shuffle scan
  if (blockIdx.x == 0) {
    __shared__ uint32_t warp_tot[kPermThreads / 32];
    const uint32_t per = (nb + kPermThreads - 1) / kPermThreads;
    const uint32_t b0 = threadIdx.x * per;
    uint32_t run = 0;
    for (uint32_t i = 0; i < per && b0 + i < nb; ++i) run += sc.count[b0 + i];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint32_t incl = run;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    if (lane == 31) warp_tot[wid] = incl;
    __syncthreads();
    uint32_t wbase = 0;
    for (int w = 0; w < wid; ++w) wbase += warp_tot[w];
    uint32_t acc = wbase + incl - run;
    for (uint32_t i = 0; i < per && b0 + i < nb; ++i) {
      sc.offset[b0 + i] = acc;
      acc += sc.count[b0 + i];
    }
    if (threadIdx.x == kPermThreads - 1) sc.offset[nb] = acc;
  }
  grid_barrier(ctrl, gridDim.x);
  // phase 3
  for (uint32_t j = tid; j < n; j += stride) {
    const uint64_t key = sc.keys[j];
    const uint32_t b = bucket_of(key, lg);
    const uint32_t pos = sc.offset[b] + atomicAdd(&sc.cursor[b], 1u);
    sc.lkey[pos] = key;
    sc.lj[pos] = j;
  }
  grid_barrier(ctrl, gridDim.x);
  // phase 4
  for (uint32_t j = tid; j < n; j += stride) {
    const uint64_t key = sc.keys[j];
    const uint32_t b = bucket_of(key, lg);
    const uint32_t lo = sc.offset[b], hi = sc.offset[b + 1];
    uint32_t r = 0;
    for (uint32_t i = lo; i < hi; ++i) {
      const uint64_t k2 = sc.lkey[i];
      r += (k2 < key) || (k2 == key && sc.lj[i] < j);
    }
    idx[lo + r] = (int64_t)((oldest + j) % cap);
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
  while ((1ull << (lg + 2)) < n) ++lg;  // nb ~ n / 4
  const uint64_t nb = 1ull << lg;
  const size_t bytes = nb * 4 * 3 + 4 + 64 + (size_t)n * (8 + 8 + 4) + 256;
  uint8_t *base = (uint8_t *)ctx_scratch(c, bytes);
  if (!base) return cudaErrorMemoryAllocation;
  PermScratch sc;
  sc.keys = (uint64_t *)base;
  sc.lkey = sc.keys + n;
  sc.count = (uint32_t *)(sc.lkey + n);
  sc.cursor = sc.count + nb;
  sc.offset = sc.cursor + nb;
  sc.lj = sc.offset + nb + 1;
  const uint64_t size = c->total < c->cap ? c->total : c->cap;
  const uint64_t oldest = (c->total - size) % c->cap;
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_permute, kPermThreads, 0);
  uint64_t grid = (n + kPermThreads - 1) / kPermThreads;
  const uint64_t cap_grid = (uint64_t)per_sm * c->coop_sms;
  if (grid > cap_grid) grid = cap_grid;
  if (grid == 0) grid = 1;
  unsigned g = (unsigned)grid;
  void *args[] = {&n, &seed, &round, &lg, &sc, (void *)&oldest,
                  (void *)&c->cap, &idx, &c->ctrl};
  return cudaLaunchCooperativeKernel((const void *)k_permute, dim3(g),
                                     dim3(kPermThreads), args, 0, s);
}

}  // namespace edp
