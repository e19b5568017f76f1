// k_llm.cu -- LLM post-training on the experience path (Appendix A): the
// group-relative advantages of GRPO (Shao et al. 2024), computed during
// ingestion, and the packed delivery of variable-length token sequences
// with a per-sequence value broadcast to their tokens.
//
// Advantages: one warp per group; fp64 sums of r and of (r - mean)^2 (two
// passes), one rounding to fp32 per output.  Packing: the batch's sequence
// lengths with each entry's source start and value (one thread each, into
// the context's scratch), a one-CTA scan of the lengths into the output
// offsets, then one CTA per sequence copies its tokens (4-byte loads and stores: neither the source
// nor the destination offset is aligned to more than a token) and writes
// the value beside each token.  Both copy kernels are HBM-bound.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kGrpoThreads = 256;
constexpr int kGrpoWarps = kGrpoThreads / 32;
constexpr int kScanThreads = 1024;
constexpr int kScanPer = 8;
constexpr int kPackThreads = 256;
constexpr int kPackUnroll = 8;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
  for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
  return v;
}

__global__ void __launch_bounds__(kGrpoThreads)
k_grpo(const float *__restrict__ r, const uint64_t *__restrict__ goff, uint32_t ng,
       float eps, float *__restrict__ adv) {
  const int lane = threadIdx.x & 31;
  pdl_wait();
  pdl_launch();
  for (uint64_t g = (uint64_t)blockIdx.x * kGrpoWarps + (threadIdx.x >> 5); g < ng;
       g += (uint64_t)gridDim.x * kGrpoWarps) {
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

// What the copy of batch entry k needs, resolved once: where its tokens
// start and the value its tokens carry.
struct PackEntry {
  uint64_t src;
  float value;
  uint32_t pad;
};

// Lengths of the batch's sequences, one thread per entry: out_off[k + 1] =
// len(idx[k]) (0 and a flag for an index out of range); out_off[0] = 0; and
// entry k's source start and value.
__global__ void __launch_bounds__(kPackThreads)
k_pack_lengths(const uint64_t *__restrict__ soff, uint64_t nseq,
               const int64_t *__restrict__ idx, uint32_t B, const float *__restrict__ sv,
               uint64_t *__restrict__ ooff, PackEntry *__restrict__ ent, Ctrl *ctrl) {
  pdl_wait();
  pdl_launch();
  const uint64_t k = (uint64_t)blockIdx.x * kPackThreads + threadIdx.x;
  if (k == 0) ooff[0] = 0;
  if (k >= B) return;
  const int64_t s = idx[k];
  uint64_t len = 0, a = 0;
  float value = 0.f;
  if (s >= 0 && (uint64_t)s < nseq) {
    a = soff[s];
    const uint64_t b = soff[s + 1];
    len = b > a ? b - a : 0;
    if (sv) value = sv[s];
  } else {
    flag(ctrl, DEVERR_INDEX, (unsigned long long)s);
  }
  ooff[k + 1] = len;
  ent[k] = PackEntry{a, value, 0u};
}

// In-place inclusive scan of out_off[1 .. B] in one CTA, in tiles of
// kScanThreads x kScanPer entries (each thread's entries loaded together):
// out_off[k] becomes the sum of the first k lengths.
__global__ void __launch_bounds__(kScanThreads)
k_pack_scan(uint32_t B, uint64_t *__restrict__ ooff, uint64_t cap, Ctrl *ctrl) {
  __shared__ uint64_t wsum[kScanThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  pdl_wait();
  pdl_launch();
  uint64_t *len = ooff + 1;
  uint64_t carry = 0;
  for (uint64_t base = 0; base < B; base += (uint64_t)kScanThreads * kScanPer) {
    const uint64_t k0 = base + (uint64_t)threadIdx.x * kScanPer;
    uint64_t v[kScanPer];
#pragma unroll
    for (int u = 0; u < kScanPer; ++u) v[u] = k0 + u < B ? len[k0 + u] : 0;
    uint64_t mine = 0;
#pragma unroll
    for (int u = 0; u < kScanPer; ++u) mine += v[u];
    uint64_t incl = mine;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t t = __shfl_up_sync(kFull, incl, o);
      if (lane >= o) incl += t;
    }
    if (lane == 31) wsum[wid] = incl;
    __syncthreads();
    if (wid == 0) {
      uint64_t w = wsum[lane];
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const uint64_t t = __shfl_up_sync(kFull, w, o);
        if (lane >= o) w += t;
      }
      wsum[lane] = w;  // inclusive prefix over warps
    }
    __syncthreads();
    uint64_t run = carry + incl - mine + (wid ? wsum[wid - 1] : 0);
#pragma unroll
    for (int u = 0; u < kScanPer; ++u) {
      run += v[u];
      if (k0 + u < B) len[k0 + u] = run;
    }
    carry += wsum[31];
    __syncthreads();  // wsum is rewritten by the next tile
  }
  if (threadIdx.x == 0 && carry > cap) flag(ctrl, DEVERR_OVERFLOW, (unsigned long long)carry);
}

// One CTA per sequence: one round trip for the entry and its offsets, then
// a thread keeps kPackUnroll loads in flight (2,048 tokens per CTA pass).
__global__ void __launch_bounds__(kPackThreads)
k_pack_gather(const int32_t *__restrict__ tokens, const PackEntry *__restrict__ ent,
              uint32_t B, int32_t *__restrict__ otok, const uint64_t *__restrict__ ooff,
              float *__restrict__ osv, uint64_t cap) {
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  for (uint32_t k = blockIdx.x; k < B; k += gridDim.x) {
    const PackEntry e = ent[k];
    const uint64_t dst = ooff[k], end = ooff[k + 1];
    if (end <= dst || dst >= cap) continue;
    const uint64_t n = min(end - dst, cap - dst);
    const int32_t *src = tokens + e.src;
    int32_t *out = otok + dst;
    for (uint64_t t0 = threadIdx.x; t0 < n; t0 += kPackThreads * kPackUnroll) {
      int32_t v[kPackUnroll];
#pragma unroll
      for (int u = 0; u < kPackUnroll; ++u) {
        const uint64_t t = t0 + u * kPackThreads;
        v[u] = t < n ? (int32_t)ld_stream(reinterpret_cast<const uint32_t *>(src + t), pol)
                     : 0;
      }
#pragma unroll
      for (int u = 0; u < kPackUnroll; ++u) {
        const uint64_t t = t0 + u * kPackThreads;
        if (t < n) {
          out[t] = v[u];
          if (osv) osv[dst + t] = e.value;
        }
      }
    }
  }
}

}  // namespace

cudaError_t launch_grpo(edp_ctx *c, const float *r, const uint64_t *goff, uint32_t ng,
                        float eps, float *adv, cudaStream_t s) {
  uint64_t blocks = (ng + kGrpoWarps - 1) / kGrpoWarps;
  if (blocks > 16ull * c->coop_sms) blocks = 16ull * c->coop_sms;
  return launch_pdl(k_grpo, dim3((unsigned)blocks), dim3(kGrpoThreads), s, r, goff, ng, eps,
                    adv);
}

cudaError_t launch_pack(edp_ctx *c, const int32_t *tokens, const uint64_t *soff,
                        uint64_t nseq, const int64_t *idx, uint32_t B, const float *sv,
                        int32_t *otok, uint64_t *ooff, float *osv, uint64_t cap,
                        cudaStream_t s) {
  PackEntry *ent = (PackEntry *)ctx_scratch(c, (size_t)B * sizeof(PackEntry));
  if (!ent) return cudaErrorMemoryAllocation;
  cudaError_t e = launch_pdl(k_pack_lengths, dim3((B + kPackThreads - 1) / kPackThreads),
                             dim3(kPackThreads), s, soff, nseq, idx, B, sv, ooff, ent, c->ctrl);
  if (e == cudaSuccess)
    e = launch_pdl(k_pack_scan, dim3(1), dim3(kScanThreads), s, B, ooff, cap, c->ctrl);
  if (e != cudaSuccess) return e;
  const unsigned grid = B < 65535u * 16u ? B : 65535u * 16u;
  return launch_pdl(k_pack_gather, dim3(grid), dim3(kPackThreads), s, tokens,
                    (const PackEntry *)ent, B, otok, (const uint64_t *)ooff, osv, cap);
}

}  // namespace edp
