// k_llm.cu -- LLM post-training on the experience path (Appendix A): the
// group-relative advantages of GRPO (Shao et al. 2024), computed during
// ingestion, and the packed delivery of variable-length token sequences
// with a per-sequence value broadcast to their tokens.
//
// Advantages: one warp per group, two warps per CTA so the groups spread
// over every SM (the fp64 pipe is narrow; eight warps on one SM queue on
// it); fp64 sums of r and of (r - mean)^2 (two passes), one rounding to fp32
// per output.  Packing: each batch entry's source start, length and value
// (one thread each, into the context's scratch) with a length sum per
// 256-entry chunk; then one CTA per sequence forms its output offset -- the
// chunk sums before its chunk plus the lengths before it in the chunk -- and
// copies its tokens (4-byte loads and stores: neither the source nor the
// destination offset is aligned to more than a token), writing the value
// beside each token.  Up to kDirectChunks chunks the gather CTAs add the
// chunk sums themselves; beyond that the last lengths CTA turns them into
// prefixes once.  The gather is HBM-bound.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kGrpoThreads = 64;
constexpr int kGrpoWarps = kGrpoThreads / 32;
constexpr int kPackThreads = 256;
constexpr uint64_t kPackWaitNs = 1000000000ull;  // bound of the gather's wait for its copy
constexpr uint32_t kDirectChunks = 256;  // chunk sums a gather CTA adds itself
static_assert(kDirectChunks <= kPackThreads, "a gather CTA adds one chunk sum per thread");

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

// Groups g = first, first + stride, ... of one warp.
__device__ __forceinline__ void grpo_groups(const float *__restrict__ r,
                                            const uint64_t *__restrict__ goff, uint32_t ng,
                                            float eps, float *__restrict__ adv,
                                            uint64_t first, uint64_t stride) {
  const int lane = threadIdx.x & 31;
  for (uint64_t g = first; g < ng; g += stride) {
    const uint64_t lo = goff[g], hi = goff[g + 1];
    if (hi <= lo) continue;
    const uint64_t n = hi - lo;
    double s1 = 0.0;
    for (uint64_t i = lo + lane; i < hi; i += 32) s1 += (double)r[i];
    const double mean = warp_sum(s1) / (double)n;
    double s2 = 0.0;
    for (uint64_t i = lo + lane; i < hi; i += 32) {
      const double d = (double)r[i] - mean;
      s2 = fma(d, d, s2);
    }
    s2 = warp_sum(s2);
    const double var = n > 1 ? s2 / (double)(n - 1) : 0.0;
    const double den = sqrt(var) + (double)eps;
    for (uint64_t i = lo + lane; i < hi; i += 32)
      adv[i] = den > 0.0 ? (float)(((double)r[i] - mean) / den) : 0.f;
  }
}

__global__ void __launch_bounds__(kGrpoThreads)
k_grpo(const float *__restrict__ r, const uint64_t *__restrict__ goff, uint32_t ng,
       float eps, float *__restrict__ adv) {
  pdl_wait();
  pdl_launch();
  grpo_groups(r, goff, ng, eps, adv, (uint64_t)blockIdx.x * kGrpoWarps + (threadIdx.x >> 5),
              (uint64_t)gridDim.x * kGrpoWarps);
}

// What the copy of batch entry k needs, resolved once: where its tokens
// start, how many there are, and the sequence (for its value; kNoSeq when
// the index is out of range).
struct PackEntry {
  uint64_t src;
  uint32_t seq;
  uint32_t len;
};
constexpr uint32_t kNoSeq = 0xffffffffu;

__device__ __forceinline__ uint64_t block_sum(uint64_t v, uint64_t *red) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  __syncthreads();  // red may still be read by a previous call
  if (lane == 0) red[wid] = v;
  __syncthreads();
  uint64_t t = 0;
#pragma unroll
  for (int w = 0; w < kPackThreads / 32; ++w) t += red[w];
  return t;
}

// One thread per batch entry: its entry (0 tokens and a flag for an index
// out of range); per CTA the sum of its 256 lengths.  With `pre` (more than
// kDirectChunks chunks) the last CTA to finish (a ticket that the context's
// ordered packed deliveries share) turns those sums into exclusive prefixes
// and resets the ticket.
// Chunk `cta` of `ncta` (the CTA's role; the fused GRPO kernel runs it
// beside the advantages).
__device__ __forceinline__ void pack_lengths_cta(const uint64_t *__restrict__ soff,
                                                 uint64_t nseq,
                                                 const int64_t *__restrict__ idx, uint32_t B,
                                                 PackEntry *__restrict__ ent,
                                                 uint64_t *__restrict__ part,
                                                 uint64_t *__restrict__ pre, uint32_t *work,
                                                 Ctrl *ctrl, uint32_t cta, uint32_t ncta) {
  __shared__ uint64_t red[kPackThreads / 32];
  __shared__ uint32_t ticket;
  const uint64_t k = (uint64_t)cta * kPackThreads + threadIdx.x;
  uint64_t len = 0;
  if (k < B) {
    const int64_t s = idx[k];
    uint64_t a = 0;
    uint32_t seq = kNoSeq;
    if (s >= 0 && (uint64_t)s < nseq) {
      a = soff[s];
      const uint64_t b = soff[s + 1];
      len = b > a ? b - a : 0;
      seq = (uint32_t)s;
    } else {
      flag(ctrl, DEVERR_INDEX, (unsigned long long)s);
    }
    ent[k] = PackEntry{a, seq, (uint32_t)len};
  }
  const uint64_t sum = block_sum(len, red);
  if (!pre) {
    if (threadIdx.x == 0) part[cta] = sum;
    return;
  }
  if (threadIdx.x == 0) {
    part[cta] = sum;
    __threadfence();
    ticket = atomicAdd(&work[0], 1u);
  }
  __syncthreads();
  if (ticket != ncta - 1) return;
  __threadfence();
  // the last CTA: exclusive prefix of the per-CTA sums, kPackThreads at a time
  uint64_t carry = 0;
  for (uint32_t base = 0; base < ncta; base += kPackThreads) {
    const uint32_t i = base + threadIdx.x;
    const uint64_t v = i < ncta ? __ldcg(&part[i]) : 0;
    uint64_t incl = v;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t t = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += t;
    }
    __syncthreads();
    if (lane == 31) red[wid] = incl;
    __syncthreads();
    uint64_t before = carry;
    for (int w = 0; w < wid; ++w) before += red[w];
    if (i < ncta) pre[i] = before + incl - v;
    uint64_t tile = 0;
#pragma unroll
    for (int w = 0; w < kPackThreads / 32; ++w) tile += red[w];
    carry += tile;
  }
  if (threadIdx.x == 0) work[0] = 0u;  // every CTA has taken its ticket
}

__global__ void __launch_bounds__(kPackThreads)
k_pack_lengths(const uint64_t *__restrict__ soff, uint64_t nseq,
               const int64_t *__restrict__ idx, uint32_t B, PackEntry *__restrict__ ent,
               uint64_t *__restrict__ part, uint64_t *__restrict__ pre, uint32_t *work,
               Ctrl *ctrl) {
  pdl_wait();
  pdl_launch();
  pack_lengths_cta(soff, nseq, idx, B, ent, part, pre, work, ctrl, blockIdx.x, gridDim.x);
}

// The GRPO step's first kernel: CTAs [0, ngc) compute the group advantages
// (two warps each, so the groups spread over the SMs), the others the
// batch's length pass, which needs no advantage (the gather reads them).
__global__ void __launch_bounds__(kPackThreads)
k_grpo_pack_lengths(const float *__restrict__ r, const uint64_t *__restrict__ goff,
                    uint32_t ng, float eps, float *__restrict__ adv, uint32_t ngc,
                    const uint64_t *__restrict__ soff, uint64_t nseq,
                    const int64_t *__restrict__ idx, uint32_t B, PackEntry *__restrict__ ent,
                    uint64_t *__restrict__ part, uint64_t *__restrict__ pre, uint32_t *work,
                    Ctrl *ctrl) {
  pdl_wait();
  pdl_launch();
  if (blockIdx.x < ngc) {
    const uint32_t w = threadIdx.x >> 5;
    if (w < kGrpoWarps)
      grpo_groups(r, goff, ng, eps, adv, (uint64_t)blockIdx.x * kGrpoWarps + w,
                  (uint64_t)ngc * kGrpoWarps);
    return;
  }
  pack_lengths_cta(soff, nseq, idx, B, ent, part, pre, work, ctrl, blockIdx.x - ngc,
                   gridDim.x - ngc);
}

// 4-byte store with the streaming (evict-first) L2 policy: the packed batch
// is written once and read by the learner, not by this kernel.
__device__ __forceinline__ void st_stream32(void *p, uint32_t v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.b32 [%0], %1, %2;"
               :: "l"(p), "r"(v), "l"(pol) : "memory");
}

// One CTA per sequence: its output offset is the prefix of its 256-entry
// chunk (from `pre`, or the chunk sums before it) plus the lengths before it
// in the chunk (one round trip and a block sum).  The tokens then move in
// chunks of up to kPackChunk: the source's 16-byte-aligned interior by one
// bulk copy into shared memory (completion on an mbarrier, waited for with a
// bound), its up to three unaligned tokens at either end by plain loads;
// the destination's aligned interior by 16-byte stores read from shared
// memory at the offset between the two alignments, its ends by 4-byte
// stores.  The per-token value is a fill with the same split, written while
// the copy is in flight.  The CTA of the last entry writes out_off[batch] =
// the total and flags an overflow.
constexpr uint32_t kPackChunk = 4096;  // tokens per bulk copy (16 KB of shared memory)
__global__ void __launch_bounds__(kPackThreads, 6)  // 36 registers, 16.5 KB: 6 CTAs per SM
k_pack_gather(const int32_t *__restrict__ tokens, const PackEntry *__restrict__ ent,
              const uint64_t *__restrict__ part, const uint64_t *__restrict__ pre, uint32_t B,
              const float *__restrict__ sv, int32_t *__restrict__ otok,
              uint64_t *__restrict__ ooff, float *__restrict__ osv, uint64_t cap, Ctrl *ctrl) {
  __shared__ uint64_t red[kPackThreads / 32];
  __shared__ alignas(16) uint32_t tbuf[kPackChunk + 8];
  __shared__ unsigned long long bar;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    mbar_init_fence();
  }
  __syncthreads();
  uint32_t uses = 0;  // completed phases of bar
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  for (uint32_t k = blockIdx.x; k < B; k += gridDim.x) {
    const uint32_t c = k / kPackThreads;
    const uint32_t j = c * kPackThreads + threadIdx.x;
    uint64_t v = j < k ? ent[j].len : 0;
    if (pre) {
      if (threadIdx.x == 0) v += pre[c];
    } else if (threadIdx.x < c) {
      v += part[threadIdx.x];  // c <= kDirectChunks = the block size
    }
    const PackEntry e = ent[k];
    const uint64_t dst = block_sum(v, red);
    if (threadIdx.x == 0) {
      ooff[k] = dst;
      if (k == B - 1) {
        ooff[B] = dst + e.len;
        if (dst + e.len > cap) flag(ctrl, DEVERR_OVERFLOW, (unsigned long long)(dst + e.len));
      }
    }
    if (e.len == 0 || dst >= cap) continue;
    const float value = osv && e.seq != kNoSeq ? __ldcg(&sv[e.seq]) : 0.f;
    const uint64_t n = min((uint64_t)e.len, cap - dst);
    const int32_t *src = tokens + e.src;
    int32_t *out = otok + dst;
    float *vout = osv ? osv + dst : nullptr;
    const uint32_t vbits = __float_as_uint(value);
    for (uint64_t c0 = 0; c0 < n; c0 += kPackChunk) {
      const uint32_t m = (uint32_t)min((uint64_t)kPackChunk, n - c0);
      const int32_t *sc = src + c0;
      // source: tokens [0, head) and [head + body, m) by plain loads, the
      // 16-byte-aligned [head, head + body) by one bulk copy; token t sits at
      // tbuf[t + shift], which puts token `head` on a 16-byte boundary
      const uint32_t hs = (uint32_t)(((16u - ((uint32_t)(uintptr_t)sc & 15u)) & 15u) >> 2);
      const uint32_t head = min(hs, m);
      const uint32_t body = (m - head) & ~3u;
      const uint32_t shift = (4u - head) & 3u;
      if (threadIdx.x == 0 && body) {
        // the previous chunk's reads of tbuf (generic proxy) come before
        // this copy's writes (async proxy)
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        mbar_arrive_tx(&bar, body * 4);
        bulk_load(&tbuf[head + shift], sc + head, body * 4, &bar, pol);
      }
      const uint32_t tail0 = head + body;
      if (threadIdx.x < head) tbuf[threadIdx.x + shift] = (uint32_t)sc[threadIdx.x];
      if (threadIdx.x < m - tail0)
        tbuf[tail0 + threadIdx.x + shift] = (uint32_t)sc[tail0 + threadIdx.x];
      // values: the same split on the destination
      if (vout) {
        float *vo = vout + c0;
        const uint32_t hv = min((uint32_t)(((16u - ((uint32_t)(uintptr_t)vo & 15u)) & 15u) >> 2), m);
        const uint32_t qv = (m - hv) >> 2;
        if (threadIdx.x < hv) st_stream32(vo + threadIdx.x, vbits, pol);
        const uint4 v4 = make_uint4(vbits, vbits, vbits, vbits);
        for (uint32_t i = threadIdx.x; i < qv; i += kPackThreads)
          st_stream(reinterpret_cast<uint4 *>(vo + hv) + i, v4, pol);
        const uint32_t tv = hv + 4 * qv;
        if (threadIdx.x < m - tv) st_stream32(vo + tv + threadIdx.x, vbits, pol);
      }
      if (body) {
        if (!mbar_wait(&bar, uses & 1u, kPackWaitNs)) {
          if (threadIdx.x == 0) flag(ctrl, DEVERR_TIMEOUT, k);
          mbar_wait(&bar, uses & 1u, kPackWaitNs);  // bounded: the copy lands first
        }
        ++uses;
      }
      __syncthreads();
      // destination: 16-byte stores of its aligned interior
      int32_t *oc = out + c0;
      const uint32_t ho = min((uint32_t)(((16u - ((uint32_t)(uintptr_t)oc & 15u)) & 15u) >> 2), m);
      const uint32_t q = (m - ho) >> 2;
      if (threadIdx.x < ho) st_stream32(oc + threadIdx.x, tbuf[threadIdx.x + shift], pol);
      for (uint32_t i = threadIdx.x; i < q; i += kPackThreads) {
        const uint32_t t = ho + 4 * i + shift;
        st_stream(reinterpret_cast<uint4 *>(oc + ho) + i,
                  make_uint4(tbuf[t], tbuf[t + 1], tbuf[t + 2], tbuf[t + 3]), pol);
      }
      const uint32_t to = ho + 4 * q;
      if (threadIdx.x < m - to) st_stream32(oc + to + threadIdx.x, tbuf[to + threadIdx.x + shift], pol);
      __syncthreads();  // tbuf is refilled by the next chunk
    }
  }
}

}  // namespace

cudaError_t launch_grpo(edp_ctx *c, const float *r, const uint64_t *goff, uint32_t ng,
                        float eps, float *adv, cudaStream_t s) {
  uint64_t blocks = (ng + kGrpoWarps - 1) / kGrpoWarps;
  if (blocks > 16ull * c->coop_sms) blocks = 16ull * c->coop_sms;
  // A plain launch: behind a large grid (the previous step's gather) an
  // early-launched k_grpo made the whole step slower (62 vs 46 us for the
  // 512 x 16 batch); its pdl_wait / pdl_launch are then no-ops.
  k_grpo<<<dim3((unsigned)blocks), dim3(kGrpoThreads), 0, s>>>(r, goff, ng, eps, adv);
  return cudaGetLastError();
}

namespace {

struct PackPlan {
  PackEntry *ent;
  uint64_t *part, *pre;
  uint32_t *work;
  uint32_t G;
};

cudaError_t pack_plan(edp_ctx *c, uint32_t B, cudaStream_t s, PackPlan *p) {
  p->G = (B + kPackThreads - 1) / kPackThreads;
  const size_t ent_bytes = ((size_t)B * sizeof(PackEntry) + 255) & ~(size_t)255;
  void *blk = nullptr;
  const cudaError_t e =
      ctx_scratch(c, ent_bytes + 2 * (size_t)p->G * sizeof(uint64_t), s, &blk);
  if (e != cudaSuccess) return e;
  uint8_t *scr = (uint8_t *)blk;
  p->ent = (PackEntry *)scr;
  p->part = (uint64_t *)(scr + ent_bytes);
  p->pre = p->G > kDirectChunks ? p->part + p->G : nullptr;
  // packed deliveries share the scratch above, so they are ordered, and one
  // ticket serves them all
  p->work = &c->ctrl->pack_ticket;
  return cudaSuccess;
}

cudaError_t launch_gather(edp_ctx *c, const PackPlan &p, const int32_t *tokens, uint32_t B,
                          const float *sv, int32_t *otok, uint64_t *ooff, float *osv,
                          uint64_t cap, cudaStream_t s) {
  const unsigned grid = B < 65535u * 16u ? B : 65535u * 16u;
  return launch_pdl(k_pack_gather, dim3(grid), dim3(kPackThreads), s, tokens,
                    (const PackEntry *)p.ent, (const uint64_t *)p.part,
                    (const uint64_t *)p.pre, B, sv, otok, ooff, osv, cap, c->ctrl);
}

}  // namespace

cudaError_t launch_pack(edp_ctx *c, const int32_t *tokens, const uint64_t *soff,
                        uint64_t nseq, const int64_t *idx, uint32_t B, const float *sv,
                        int32_t *otok, uint64_t *ooff, float *osv, uint64_t cap,
                        cudaStream_t s) {
  PackPlan p;
  cudaError_t e = pack_plan(c, B, s, &p);
  if (e != cudaSuccess) return e;
  e = launch_pdl(k_pack_lengths, dim3(p.G), dim3(kPackThreads), s, soff, nseq,
                             idx, B, p.ent, p.part, p.pre, p.work, c->ctrl);
  if (e != cudaSuccess) return e;
  return launch_gather(c, p, tokens, B, sv, otok, ooff, osv, cap, s);
}

cudaError_t launch_grpo_pack(edp_ctx *c, const float *r, const uint64_t *goff, uint32_t ng,
                             float eps, float *adv, const int32_t *tokens,
                             const uint64_t *soff, uint64_t nseq, const int64_t *idx,
                             uint32_t B, int32_t *otok, uint64_t *ooff, float *osv,
                             uint64_t cap, cudaStream_t s) {
  PackPlan p;
  cudaError_t e = pack_plan(c, B, s, &p);
  if (e != cudaSuccess) return e;
  uint64_t ngc = (ng + kGrpoWarps - 1) / kGrpoWarps;
  if (ngc > 16ull * c->coop_sms) ngc = 16ull * c->coop_sms;
  // a plain launch, as for k_grpo
  k_grpo_pack_lengths<<<dim3((unsigned)(ngc + p.G)), dim3(kPackThreads), 0, s>>>(
      r, goff, ng, eps, adv, (uint32_t)ngc, soff, nseq, idx, B, p.ent, p.part, p.pre, p.work,
      c->ctrl);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  return launch_gather(c, p, tokens, B, adv, otok, ooff, osv, cap, s);
}

}  // namespace edp
