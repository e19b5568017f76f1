// k_ring.cu -- ingestion kernels: ring scatter of payload rows, metadata and
// priority leaves, two-tier demotion, and the host-link read probe.
//
// Ingestion inserts transitions into the persistent buffer and maintains the
// indices and metadata used for sampling and eviction (Sec. 2.2, off-policy
// ingestion).  Payload rows are moved with 16-byte vector loads and stores,
// several loads in flight per thread; the ring index arithmetic is done once
// per row, never per element.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr int kCopyThreads = 256;
constexpr int kCopyUnroll = 4;

// Copy of up to three contiguous runs of 16-byte words (a range of ring
// rows splits where the source or the destination wraps): a flat
// grid-stride loop, kCopyFlat words in flight per thread, so the copy is
// one stream of full 16-byte accesses whatever the row size.  src may be
// page-locked host memory (mapped).  With wait_first the kernel waits for
// the preceding kernel before it reads or writes anything; otherwise it
// starts at once -- allowed only right behind a kernel of the same call that
// waited on its own predecessor, so the rows it overwrites are no longer
// read -- and waits at its end, so it never completes before that kernel.
constexpr int kCopyFlat = 8;
constexpr int kCopyCtasPerSm = 64;
struct CopyRuns {
  const uint4 *src[3];
  uint4 *dst[3];
  uint64_t end[3];  // cumulative word counts; unused runs repeat the total
};

// Tiles of kThr * kCopyFlat words of the runs, CTA `cta` of `ncta`: each
// warp-wide access moves 512 contiguous bytes, a CTA's loads cover one
// contiguous tile.
template <int kThr>
__device__ __forceinline__ void copy_tiles(const CopyRuns &r, uint64_t cta, uint64_t ncta) {
  const uint64_t total = r.end[2];  // unused runs repeat the last end
  constexpr uint64_t kTile = (uint64_t)kThr * kCopyFlat;  // words per tile
  const uint64_t tiles = (total + kTile - 1) / kTile;
  for (uint64_t t = cta; t < tiles; t += ncta) {
    const uint64_t i0 = t * kTile + threadIdx.x;
    uint4 v[kCopyFlat];
#pragma unroll
    for (int u = 0; u < kCopyFlat; ++u) {
      const uint64_t i = i0 + (uint64_t)u * kThr;
      if (i < total) {
        // run of word i, selected without indexing the parameter array
        // (which would place it in local memory)
        const bool g1 = i >= r.end[0], g2 = i >= r.end[1];
        const uint64_t o = g2 ? i - r.end[1] : (g1 ? i - r.end[0] : i);
        v[u] = (g2 ? r.src[2] : (g1 ? r.src[1] : r.src[0]))[o];
      }
    }
#pragma unroll
    for (int u = 0; u < kCopyFlat; ++u) {
      const uint64_t i = i0 + (uint64_t)u * kThr;
      if (i < total) {
        const bool g1 = i >= r.end[0], g2 = i >= r.end[1];
        const uint64_t o = g2 ? i - r.end[1] : (g1 ? i - r.end[0] : i);
        (g2 ? r.dst[2] : (g1 ? r.dst[1] : r.dst[0]))[o] = v[u];
      }
    }
  }
}

__global__ void __launch_bounds__(kCopyThreads)
k_copy_flat(CopyRuns r, int wait_first) {
  if (wait_first) pdl_wait();
  pdl_launch();
  copy_tiles<kCopyThreads>(r, blockIdx.x, gridDim.x);
  if (!wait_first) pdl_wait();
}

// The runs of rows (src_first + j) mod src_cap -> (dst_first + j) mod
// dst_cap, j < n: contiguous between the wrap points of either side.
CopyRuns row_runs(uint8_t *dst, uint64_t dst_cap, uint64_t dst_first, const uint8_t *src,
                  uint64_t src_cap, uint64_t src_first, uint64_t n, uint64_t row_bytes) {
  uint64_t cut[4] = {0, n, n, n};
  int nc = 1;
  const uint64_t jd = dst_cap - dst_first, js = src_cap - src_first;
  for (uint64_t j : {jd < js ? jd : js, jd < js ? js : jd})
    if (j > cut[nc - 1] && j < n) cut[nc++] = j;
  cut[nc] = n;
  CopyRuns r{};
  uint64_t acc = 0;
  for (int g = 0; g < nc; ++g) {
    const uint64_t j0 = cut[g];
    r.src[g] = reinterpret_cast<const uint4 *>(src + ((src_first + j0) % src_cap) * row_bytes);
    r.dst[g] = reinterpret_cast<uint4 *>(dst + ((dst_first + j0) % dst_cap) * row_bytes);
    acc += (cut[g + 1] - j0) * (row_bytes / 16);
    r.end[g] = acc;
  }
  for (int g = nc; g < 3; ++g) r.end[g] = acc;
  return r;
}

int sm_count() {
  int dev = 0, sms = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  return sms > 0 ? sms : 1;
}

// Swap rows through HBM: HBM row (first + j) mod hbm_cap moves to host row
// (first + j) mod host_cap and source row j takes its place.  One thread
// handles one 16-byte chunk in all three rows, reading the old HBM value
// before writing the new one, so no other thread's order matters.  The
// host-link traffic goes both ways at once (source rows in, demoted rows
// out), which a demotion followed by a copy would serialise.
__global__ void __launch_bounds__(kCopyThreads)
k_swap_rows(uint8_t *__restrict__ hbm, uint64_t hbm_cap, uint8_t *__restrict__ host,
            uint64_t host_cap, const uint8_t *__restrict__ src, uint64_t first,
            uint64_t n, uint32_t cpr) {
  const uint64_t row_bytes = (uint64_t)cpr * 16u;
  for (uint64_t j = blockIdx.y; j < n; j += gridDim.y) {
    uint4 *h = reinterpret_cast<uint4 *>(hbm + ((first + j) % hbm_cap) * row_bytes);
    uint4 *c = reinterpret_cast<uint4 *>(host + ((first + j) % host_cap) * row_bytes);
    const uint4 *s = reinterpret_cast<const uint4 *>(src + j * row_bytes);
    const uint32_t step = gridDim.x * kCopyThreads * kCopyUnroll;
    for (uint32_t w0 = blockIdx.x * kCopyThreads * kCopyUnroll + threadIdx.x;
         w0 < cpr; w0 += step) {
      uint4 old_[kCopyUnroll], new_[kCopyUnroll];
#pragma unroll
      for (int u = 0; u < kCopyUnroll; ++u) {
        const uint32_t w = w0 + u * kCopyThreads;
        if (w < cpr) {
          old_[u] = h[w];
          new_[u] = s[w];
        }
      }
#pragma unroll
      for (int u = 0; u < kCopyUnroll; ++u) {
        const uint32_t w = w0 + u * kCopyThreads;
        if (w < cpr) {
          c[w] = old_[u];
          h[w] = new_[u];
        }
      }
    }
  }
}

cudaError_t swap_rows(uint8_t *hbm, uint64_t hbm_cap, uint8_t *host, uint64_t host_cap,
                      const uint8_t *src, uint64_t first, uint64_t n,
                      uint64_t row_bytes, cudaStream_t s) {
  if (!n) return cudaSuccess;
  const uint32_t cpr = (uint32_t)(row_bytes / 16);
  uint32_t gx = (cpr + kCopyThreads * kCopyUnroll - 1) / (kCopyThreads * kCopyUnroll);
  if (gx > 64) gx = 64;
  const uint32_t gy = n < 65535 ? (uint32_t)n : 65535u;
  k_swap_rows<<<dim3(gx, gy), kCopyThreads, 0, s>>>(hbm, hbm_cap, host, host_cap, src,
                                                   first, n, cpr);
  return cudaGetLastError();
}

// Rows (src_first + j) mod src_cap -> (dst_first + j) mod dst_cap for
// j < n, as the contiguous runs between the wrap points of either side.
cudaError_t copy_rows(uint8_t *dst, uint64_t dst_cap, uint64_t dst_first,
                      const uint8_t *src, uint64_t src_cap, uint64_t src_first,
                      uint64_t n, uint64_t row_bytes, cudaStream_t s, bool wait_first) {
  if (!n) return cudaSuccess;
  const CopyRuns r = row_runs(dst, dst_cap, dst_first, src, src_cap, src_first, n, row_bytes);
  const uint64_t acc = r.end[2];
  uint64_t blocks = (acc + (uint64_t)kCopyThreads * kCopyFlat - 1) / ((uint64_t)kCopyThreads * kCopyFlat);
  const uint64_t most = (uint64_t)kCopyCtasPerSm * sm_count();
  if (blocks > most) blocks = most;
  return launch_pdl(k_copy_flat, dim3((unsigned)blocks), dim3(kCopyThreads), s, r,
                    wait_first ? 1 : 0);
}

// Metadata of n new transitions at logical ids total.. and, for PER, their
// leaves.  With `defer` the newest transition's leaf stays 0 and its
// priority waits in ctrl->pending_q; the previous newest (id total-1) gets
// its pending priority now -- unless this insertion overwrites its slot.
struct MetaArgs {
  int32_t *action;
  float *reward;
  uint8_t *done;
  const int32_t *s_action;
  const float *s_reward;
  const uint8_t *s_done;
  uint32_t *leaves;
  const uint32_t *q;
  Ctrl *ctrl;
  uint64_t cap, total, n;
  int defer;
};

// Transitions j = j0, j0 + stride, ... of the insertion, kMetaBatch at a
// time: the batch's source loads are all issued before its stores (a store
// to the ring could alias a source as far as the compiler knows, so loads
// interleaved with stores would each wait a round trip).
constexpr int kMetaBatch = 4;
__device__ __forceinline__ void ingest_meta_range(const MetaArgs &a, uint64_t j0,
                                                  uint64_t stride) {
  uint32_t qdefault = 0;
  if (a.leaves && !a.q) qdefault = a.ctrl->max_q;
  uint32_t qmax_local = 0;  // one atomic per warp, not per transition
  for (uint64_t jb = j0; jb < a.n; jb += kMetaBatch * stride) {
    int32_t act[kMetaBatch];
    float rew[kMetaBatch];
    uint8_t dn[kMetaBatch];
    uint32_t qs[kMetaBatch];
#pragma unroll
    for (int b = 0; b < kMetaBatch; ++b) {
      const uint64_t j = jb + b * stride;
      const bool in = j < a.n;
      act[b] = in && a.s_action ? a.s_action[j] : 0;
      rew[b] = in && a.s_reward ? a.s_reward[j] : 0.f;
      dn[b] = in && a.s_done ? a.s_done[j] : (uint8_t)0;
      qs[b] = in && a.q ? a.q[j] : qdefault;
    }
#pragma unroll
    for (int b = 0; b < kMetaBatch; ++b) {
      const uint64_t j = jb + b * stride;
      if (j >= a.n) break;
      const uint64_t m = (a.total + j) % a.cap;
      if (a.action) a.action[m] = act[b];
      if (a.reward) a.reward[m] = rew[b];
      if (a.done) a.done[m] = dn[b];
      if (a.leaves) {
        const uint32_t qj = qs[b];
        if (a.q) qmax_local = max(qmax_local, qj);
        if (a.defer) {
          a.leaves[m] = (j == a.n - 1) ? 0u : qj;
          if (j == 0) {
            // only this thread touches pending_q and the previous newest leaf
            if (a.total >= 1 && a.n < a.cap)
              a.leaves[(a.total - 1) % a.cap] = a.ctrl->pending_q;
            a.ctrl->pending_q = a.q ? a.q[a.n - 1] : qdefault;
          }
        } else {
          a.leaves[m] = qj;
        }
      }
    }
  }
  if (a.leaves && a.q) {
#pragma unroll
    for (int o = 16; o; o >>= 1)
      qmax_local = max(qmax_local, __shfl_xor_sync(0xffffffffu, qmax_local, o));
    if ((threadIdx.x & 31) == 0 && qmax_local) atomicMax(&a.ctrl->max_q, qmax_local);
  }
}

__global__ void k_ingest_meta(MetaArgs a) {
  pdl_wait();
  pdl_launch();
  ingest_meta_range(a, blockIdx.x * (uint64_t)blockDim.x + threadIdx.x,
                    (uint64_t)gridDim.x * blockDim.x);
}

// One insertion in one launch (replay rings: a single HBM tier, at most
// kFusedMaxRows rows).  CTA 0 writes the metadata and leaves, then refreshes
// the tree above them level by level (a CTA barrier between levels, so each
// level reads the sums written below it); the other CTAs copy the payload
// rows (obs, then tokens).  Nothing of the two parts reads what the other
// writes, so the metadata chain runs beside the copy.
constexpr int kFusedThreads = 1024;
constexpr uint64_t kFusedMaxRows = 16384;

struct TreeRefresh {
  uint64_t *level[kMaxDepth];  // level d: 32^d sums
  uint32_t *leaves;
  uint32_t depth;
  // nodes of level d to recompute: [a0, a0 + n0) and [a1, a1 + n1)
  uint64_t a0[kMaxDepth], n0[kMaxDepth], a1[kMaxDepth], n1[kMaxDepth];
};

__global__ void __launch_bounds__(kFusedThreads, 1)
k_ingest_fused(CopyRuns obs, CopyRuns tok, MetaArgs meta, TreeRefresh t) {
  pdl_wait();
  pdl_launch();
  if (blockIdx.x != 0) {
    copy_tiles<kFusedThreads>(obs, blockIdx.x - 1, gridDim.x - 1);
    copy_tiles<kFusedThreads>(tok, blockIdx.x - 1, gridDim.x - 1);
    return;
  }
  ingest_meta_range(meta, threadIdx.x, kFusedThreads);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  constexpr int kWarps = kFusedThreads / 32;
#pragma unroll
  for (int d = kMaxDepth - 1; d >= 0; --d) {  // constant indices into t
    if ((uint32_t)d >= t.depth) continue;
    __syncthreads();  // the level below (or the leaves) is written
    const bool leaves_below = (uint32_t)d + 1 == t.depth;
    const uint64_t n = t.n0[d] + t.n1[d];
    for (uint64_t w = warp; w < n; w += kWarps) {
      const uint64_t node = w < t.n0[d] ? t.a0[d] + w : t.a1[d] + (w - t.n0[d]);
      const uint64_t c = node * kFanout + lane;
      uint64_t v = leaves_below ? (uint64_t)__ldcg(t.leaves + c)
                                : __ldcg(t.level[d + 1 < kMaxDepth ? d + 1 : d] + c);
#pragma unroll
      for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
      if (lane == 0) t.level[d][node] = v;
    }
  }
}

// Host-link probe: stream n16 16-byte words (page-locked host memory,
// device-mapped) through the SMs, xor-folding them so no load is dead.
__global__ void k_probe_read(const uint4 *__restrict__ src, uint64_t n16,
                             unsigned long long *fold) {
  uint4 acc = make_uint4(0, 0, 0, 0);
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  uint64_t i = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x;
  for (; i + 3 * stride < n16; i += 4 * stride) {
    const uint4 a = src[i], b = src[i + stride], c = src[i + 2 * stride],
                d = src[i + 3 * stride];
    acc.x ^= a.x ^ b.x ^ c.x ^ d.x;
    acc.y ^= a.y ^ b.y ^ c.y ^ d.y;
    acc.z ^= a.z ^ b.z ^ c.z ^ d.z;
    acc.w ^= a.w ^ b.w ^ c.w ^ d.w;
  }
  for (; i < n16; i += stride) {
    const uint4 a = src[i];
    acc.x ^= a.x;
    acc.y ^= a.y;
    acc.z ^= a.z;
    acc.w ^= a.w;
  }
  unsigned long long v = ((unsigned long long)(acc.x ^ acc.z) << 32) | (acc.y ^ acc.w);
#pragma unroll
  for (int o = 16; o; o >>= 1) v ^= __shfl_xor_sync(0xffffffffu, v, o);
  if ((threadIdx.x & 31) == 0 && v) atomicXor(fold, v);
}

}  // namespace

cudaError_t launch_copy_rows(uint8_t *dst, uint64_t dst_cap, uint64_t first,
                             const uint8_t *src, uint64_t n, uint64_t row_bytes,
                             cudaStream_t s, bool wait_first) {
  return copy_rows(dst, dst_cap, first, src, ~0ull, 0, n, row_bytes, s, wait_first);
}

namespace {
MetaArgs meta_args(edp_ctx *c, const edp_fields *f, uint64_t n, const uint32_t *q) {
  MetaArgs a{};
  a.action = c->st.action;
  a.reward = c->st.reward;
  a.done = c->st.done;
  a.s_action = f->action;
  a.s_reward = f->reward;
  a.s_done = f->done;
  a.leaves = c->leaves;
  a.q = q;
  a.ctrl = c->ctrl;
  a.cap = c->cap;
  a.total = c->total;
  a.n = n;
  a.defer = c->defer;
  return a;
}
}  // namespace

cudaError_t launch_ingest_meta(edp_ctx *c, const edp_fields *f, uint64_t n,
                               const uint32_t *q, cudaStream_t s) {
  if (!c->st.action && !c->st.reward && !c->st.done && !c->leaves)
    return cudaSuccess;
  const int threads = 256;
  uint64_t blocks = (n + threads - 1) / threads;
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(k_ingest_meta, dim3((unsigned)blocks), dim3(threads), s,
                    meta_args(c, f, n, q));
}

bool ingest_fusable(const edp_ctx *c, uint64_t n) {
  return c->cap_c == 0 && n <= kFusedMaxRows;
}

cudaError_t launch_ingest_fused(edp_ctx *c, const edp_fields *f, uint64_t n,
                                const uint32_t *q, uint64_t tree_first, uint64_t tree_count,
                                cudaStream_t s) {
  const uint64_t first = c->total % c->cap_h;
  const CopyRuns obs = row_runs(c->st.obs, c->cap_h, first, f->obs, ~0ull, 0, n, c->obs_bytes);
  CopyRuns tok{};
  if (c->tok_bytes)
    tok = row_runs((uint8_t *)c->st.tokens, c->cap_h, first, (const uint8_t *)f->tokens, ~0ull,
                   0, n, c->tok_bytes);
  TreeRefresh t{};
  if (c->depth && tree_count) {
    TreeRanges tr;
    tree_ranges(c, tree_first, tree_count, &tr);
    t.depth = c->depth;
    t.leaves = c->leaves;
    for (uint32_t d = 0; d < c->depth; ++d) {
      t.level[d] = c->level[d];
      t.a0[d] = tr.a0[d];
      t.n0[d] = tr.n0[d];
      t.a1[d] = tr.a1[d];
      t.n1[d] = tr.n1[d];
    }
  }
  const uint64_t words = obs.end[2] + tok.end[2];
  uint64_t blocks = (words + (uint64_t)kFusedThreads * kCopyFlat - 1) /
                    ((uint64_t)kFusedThreads * kCopyFlat);
  const uint64_t most = 2ull * sm_count();
  if (blocks > most) blocks = most;
  return launch_pdl(k_ingest_fused, dim3((unsigned)(blocks + 1)), dim3(kFusedThreads), s, obs,
                    tok, meta_args(c, f, n, q), t);
}

// Two-tier demotion: payload of ids [first_id, first_id+n) moves from HBM
// slot L mod cap_h to host slot L mod cap_c, before new payload overwrites
// those HBM slots (same stream).
cudaError_t launch_demote(edp_ctx *c, uint64_t first_id, uint64_t n,
                          cudaStream_t s) {
  cudaError_t e = copy_rows(c->st.host_obs, c->cap_c, first_id % c->cap_c,
                            c->st.obs, c->cap_h, first_id % c->cap_h, n,
                            c->obs_bytes, s, true);
  if (e == cudaSuccess && c->tok_bytes)
    e = copy_rows((uint8_t *)c->st.host_tokens, c->cap_c, first_id % c->cap_c,
                  (const uint8_t *)c->st.tokens, c->cap_h, first_id % c->cap_h,
                  n, c->tok_bytes, s, true);
  return e;
}

cudaError_t launch_swap(edp_ctx *c, uint64_t first_id, const uint8_t *obs,
                        const int32_t *tokens, uint64_t n, cudaStream_t s) {
  cudaError_t e = swap_rows(c->st.obs, c->cap_h, c->st.host_obs, c->cap_c, obs,
                            first_id, n, c->obs_bytes, s);
  if (e == cudaSuccess && c->tok_bytes)
    e = swap_rows((uint8_t *)c->st.tokens, c->cap_h, (uint8_t *)c->st.host_tokens,
                  c->cap_c, (const uint8_t *)tokens, first_id, n, c->tok_bytes, s);
  return e;
}

// ---- migration between placements (Sec. 5.3, Alg. 2) ---------------------
// Where the payload row of logical id L lives in a ring with `total`
// insertions: the newest min(total, cap_h) ids in HBM at L mod cap_h, older
// ones in the host tier at L mod cap_c.
struct TierView {
  uint8_t *hbm;
  uint8_t *host;
  uint64_t cap_h, cap_c, total, row;
};

__device__ __forceinline__ uint8_t *tier_row(const TierView &v, uint64_t L) {
  const uint64_t in_hbm = v.total < v.cap_h ? v.total : v.cap_h;
  if (L >= v.total - in_hbm) return v.hbm + (L % v.cap_h) * v.row;
  return v.host + (L % v.cap_c) * v.row;
}

// Rows of source ids [L0, L0 + n), renumbered 0 .. n-1 in dst, from their
// place in src to their place in dst; every direction (HBM or host to HBM
// or host) runs in the same launch.
__global__ void __launch_bounds__(kCopyThreads)
k_migrate_rows(TierView src, TierView dst, uint64_t L0, uint64_t n) {
  const uint32_t cpr = (uint32_t)(src.row / 16);
  for (uint64_t j = blockIdx.y; j < n; j += gridDim.y) {
    const uint4 *s = reinterpret_cast<const uint4 *>(tier_row(src, L0 + j));
    uint4 *d = reinterpret_cast<uint4 *>(tier_row(dst, j));
    const uint32_t step = gridDim.x * kCopyThreads * kCopyUnroll;
    for (uint32_t w0 = blockIdx.x * kCopyThreads * kCopyUnroll + threadIdx.x; w0 < cpr;
         w0 += step) {
      uint4 v[kCopyUnroll];
#pragma unroll
      for (int u = 0; u < kCopyUnroll; ++u) {
        const uint32_t w = w0 + u * kCopyThreads;
        if (w < cpr) v[u] = s[w];
      }
#pragma unroll
      for (int u = 0; u < kCopyUnroll; ++u) {
        const uint32_t w = w0 + u * kCopyThreads;
        if (w < cpr) d[w] = v[u];
      }
    }
  }
}

// Metadata and priority leaves of source ids [L0, L0 + n): slot
// (L0 + j) mod cap_s in src, j mod cap_d in dst.
__global__ void k_migrate_meta(const int32_t *sa, const float *sr, const uint8_t *sd,
                               const uint32_t *sl, uint64_t cap_s, int32_t *da, float *dr,
                               uint8_t *dd, uint32_t *dl, uint64_t cap_d, uint64_t L0,
                               uint64_t n) {
  for (uint64_t j = blockIdx.x * (uint64_t)blockDim.x + threadIdx.x; j < n;
       j += (uint64_t)gridDim.x * blockDim.x) {
    const uint64_t ms = (L0 + j) % cap_s, md = j % cap_d;
    if (da) da[md] = sa ? sa[ms] : 0;
    if (dr) dr[md] = sr ? sr[ms] : 0.f;
    if (dd) dd[md] = sd ? sd[ms] : (uint8_t)0;
    if (dl) dl[md] = sl ? sl[ms] : 0u;
  }
}

cudaError_t migrate_payload(const TierView &s, const TierView &d, uint64_t L0, uint64_t n,
                            cudaStream_t st) {
  if (!n) return cudaSuccess;
  const uint32_t cpr = (uint32_t)(s.row / 16);
  uint32_t gx = (cpr + kCopyThreads * kCopyUnroll - 1) / (kCopyThreads * kCopyUnroll);
  if (gx > 64) gx = 64;
  const uint32_t gy = n < 65535 ? (uint32_t)n : 65535u;
  k_migrate_rows<<<dim3(gx, gy), kCopyThreads, 0, st>>>(s, d, L0, n);
  return cudaGetLastError();
}

cudaError_t launch_migrate(const edp_ctx *src, edp_ctx *dst, uint64_t L0, uint64_t n,
                           cudaStream_t st) {
  TierView s{src->st.obs, src->st.host_obs, src->cap_h, src->cap_c ? src->cap_c : 1,
             src->total, src->obs_bytes};
  TierView d{dst->st.obs, dst->st.host_obs, dst->cap_h, dst->cap_c ? dst->cap_c : 1, n,
             dst->obs_bytes};
  cudaError_t e = migrate_payload(s, d, L0, n, st);
  if (e == cudaSuccess && src->tok_bytes) {
    s.hbm = (uint8_t *)src->st.tokens;
    s.host = (uint8_t *)src->st.host_tokens;
    s.row = src->tok_bytes;
    d.hbm = (uint8_t *)dst->st.tokens;
    d.host = (uint8_t *)dst->st.host_tokens;
    d.row = dst->tok_bytes;
    e = migrate_payload(s, d, L0, n, st);
  }
  if (e != cudaSuccess || !n) return e;
  const int threads = 256;
  uint64_t blocks = (n + threads - 1) / threads;
  if (blocks > 4096) blocks = 4096;
  k_migrate_meta<<<(unsigned)blocks, threads, 0, st>>>(
      src->st.action, src->st.reward, src->st.done, src->leaves, src->cap, dst->st.action,
      dst->st.reward, dst->st.done, dst->leaves, dst->cap, L0, n);
  return cudaGetLastError();
}

cudaError_t launch_copy_rows_to_host(edp_ctx *c, const uint8_t *obs,
                                     const int32_t *tokens, uint64_t src_row,
                                     uint64_t first_id, uint64_t n,
                                     cudaStream_t s) {
  cudaError_t e = copy_rows(c->st.host_obs, c->cap_c, first_id % c->cap_c,
                            obs + src_row * c->obs_bytes, ~0ull, 0, n,
                            c->obs_bytes, s, true);
  if (e == cudaSuccess && c->tok_bytes)
    e = copy_rows((uint8_t *)c->st.host_tokens, c->cap_c, first_id % c->cap_c,
                  (const uint8_t *)tokens + src_row * c->tok_bytes, ~0ull, 0, n,
                  c->tok_bytes, s, true);
  return e;
}

cudaError_t launch_probe_read(const void *src, uint64_t bytes, uint64_t *fold,
                              cudaStream_t s) {
  int sms = 0, dev = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  k_probe_read<<<sms * 4, 512, 0, s>>>((const uint4 *)src, bytes / 16,
                                       (unsigned long long *)fold);
  return cudaGetLastError();
}

}  // namespace edp
