// k_llm.cu -- LLM post-training on the experience path (Appendix A): the
// group-relative advantages of GRPO (Shao et al. 2024), computed during
// ingestion, and the packed delivery of variable-length token sequences
// with a per-sequence value broadcast to their tokens.
//
// Advantages: one warp per group; fp64 sums of r and of (r - mean)^2 (two
// passes), one rounding to fp32 per output.  Packing: a one-CTA scan of the
// batch's sequence lengths writes the output offsets, then one CTA per
// sequence copies its tokens (4-byte loads and stores: neither the source
// nor the destination offset is aligned to more than a token) and writes
// the value beside each token.  Both copy kernels are HBM-bound.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kGrpoThreads = 256;
constexpr int kGrpoWarps = kGrpoThreads / 32;
constexpr int kScanThreads = 1024;
constexpr int kPackThreads = 256;
constexpr int kPackUnroll = 4;

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

// length of batch entry k, or 0 (and a flag) for an index out of range
__device__ __forceinline__ uint64_t seq_len(const uint64_t *soff, uint64_t nseq,
                                            const int64_t *idx, uint32_t k, Ctrl *ctrl) {
  const int64_t s = idx[k];
  if (s < 0 || (uint64_t)s >= nseq) {
    if (ctrl) flag(ctrl, DEVERR_INDEX, (unsigned long long)s);
    return 0;
  }
  const uint64_t a = soff[s], b = soff[s + 1];
  return b > a ? b - a : 0;
}

// Exclusive scan of the batch's lengths in one CTA: thread t owns entries
// [t per, (t+1) per); out_off[batch] = the total.
__global__ void __launch_bounds__(kScanThreads)
k_pack_offsets(const uint64_t *__restrict__ soff, uint64_t nseq,
               const int64_t *__restrict__ idx, uint32_t B, uint64_t *__restrict__ ooff,
               uint64_t cap, Ctrl *ctrl) {
  __shared__ uint64_t wsum[kScanThreads / 32];
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  pdl_wait();
  pdl_launch();
  const uint32_t per = (B + kScanThreads - 1) / kScanThreads;
  const uint32_t k0 = threadIdx.x * per, k1 = min(B, k0 + per);
  uint64_t mine = 0;
  for (uint32_t k = k0; k < k1; ++k) mine += seq_len(soff, nseq, idx, k, nullptr);
  // inclusive warp scan, then across warps
  uint64_t incl = mine;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint64_t v = __shfl_up_sync(kFull, incl, o);
    if (lane >= o) incl += v;
  }
  if (lane == 31) wsum[wid] = incl;
  __syncthreads();
  if (wid == 0) {
    uint64_t w = wsum[lane];
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint64_t v = __shfl_up_sync(kFull, w, o);
      if (lane >= o) w += v;
    }
    wsum[lane] = w;  // inclusive prefix over warps
  }
  __syncthreads();
  uint64_t run = incl - mine + (wid ? wsum[wid - 1] : 0);
  for (uint32_t k = k0; k < k1; ++k) {
    ooff[k] = run;
    run += seq_len(soff, nseq, idx, k, ctrl);
  }
  if (threadIdx.x == kScanThreads - 1) {
    ooff[B] = run;
    if (run > cap) flag(ctrl, DEVERR_OVERFLOW, (unsigned long long)run);
  }
}

__global__ void __launch_bounds__(kPackThreads)
k_pack_gather(const int32_t *__restrict__ tokens, const uint64_t *__restrict__ soff,
              uint64_t nseq, const int64_t *__restrict__ idx, uint32_t B,
              const float *__restrict__ sv, int32_t *__restrict__ otok,
              const uint64_t *__restrict__ ooff, float *__restrict__ osv, uint64_t cap) {
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  for (uint32_t k = blockIdx.x; k < B; k += gridDim.x) {
    const int64_t s = idx[k];
    if (s < 0 || (uint64_t)s >= nseq) continue;  // flagged by the scan
    const uint64_t a = soff[s], b = soff[s + 1];
    const uint64_t dst = ooff[k];
    if (b <= a || dst >= cap) continue;
    const uint64_t n = min(b - a, cap - dst);
    const int32_t *src = tokens + a;
    int32_t *out = otok + dst;
    const float value = sv ? sv[s] : 0.f;
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
          if (osv) osv[dst + t] = value;
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
  cudaError_t e = launch_pdl(k_pack_offsets, dim3(1), dim3(kScanThreads), s, soff, nseq, idx,
                             B, ooff, cap, c->ctrl);
  if (e != cudaSuccess) return e;
  const unsigned grid = B < 65535u * 16u ? B : 65535u * 16u;
  return launch_pdl(k_pack_gather, dim3(grid), dim3(kPackThreads), s, tokens, soff, nseq, idx,
                    B, sv, otok, (const uint64_t *)ooff, osv, cap);
}

}  // namespace edp
