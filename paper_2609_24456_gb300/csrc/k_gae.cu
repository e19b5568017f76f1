// k_gae.cu -- generalized advantage estimation with global advantage
// normalisation (Schulman et al., ICLR'16; the return / advantage and
// normalisation steps of on-policy ingestion, Sec. 2.2).
//
//   delta_t = r_t + gamma V_{t+1} (1 - d_t) - V_t
//   A_t = delta_t + c_t A_{t+1},  c_t = gamma lambda (1 - d_t),  A_T = 0
//
// The recurrence is a composition of affine maps x -> b + a x, which is
// associative, so one warp scans one environment's T steps in parallel:
// each lane composes the maps of J consecutive steps, a warp-shuffle suffix
// scan composes lanes (5 levels), and each lane then replays its own steps
// from the value handed over by its right neighbour.  Chunks of 32*J steps
// are processed from the end of the rollout backwards, carrying A across.
//
// Arithmetic: GB300's fp64 pipe is narrow (a dependent fp64 FMA costs ~64
// cycles, fp32 ~4), so the scan -- and each lane's sums of A and A^2 over an
// environment -- run in double-float arithmetic -- a value
// is an unevaluated pair hi + lo of fp32 numbers, combined with the
// error-free transformations TwoSum (Knuth) and TwoProd via FMA (Dekker),
// as in the double-double arithmetic of Hida, Li and Bailey -- which keeps
// ~44 significant bits (relative error ~2^-44 per operation); gamma and
// gamma*lambda enter as pairs split from fp64.  Only the mean / variance
// reduction and the normalisation use fp64.  Outputs are rounded to fp32.
//
// Two kernels chained with programmatic dependent launch: the scan writes A,
// the returns and per-CTA fp64 sums of A and A^2; the normalisation kernel
// forms mean and the unbiased standard deviation (every CTA reduces the
// partials in the same fixed order, so all agree bit for bit) and writes
// the normalised values, one thread per element.  With the environments
// sharded over several ranks, the scan's sums are reduced to this rank's
// (n, sum A, sum A^2) instead (k_gae_stats), the caller sums those over the
// ranks, and the normalisation reads the totals.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kJ = 4;          // steps per lane per chunk
constexpr int kGaeWarps = 4;   // environments per CTA
constexpr int kGaeThreads = kGaeWarps * 32;
constexpr int kNormThreads = 256;

__device__ __forceinline__ df df_shfl_down(df a, int o) {
  return {__shfl_down_sync(kFull, a.hi, o), __shfl_down_sync(kFull, a.lo, o)};
}
// One environment's scan (one warp): writes its advantages and returns and
// adds this lane's A and A^2 to s1, s2.
__device__ __forceinline__ void gae_env(const float *__restrict__ r,
                                        const float *__restrict__ v,
                                        const uint8_t *__restrict__ d, uint32_t T, uint32_t E,
                                        uint32_t e, df g, df gl, float *__restrict__ A_out,
                                        float *__restrict__ ret, double &s1, double &s2) {
  const int lane = threadIdx.x & 31;
  const df one = {1.f, 0.f}, zero = {0.f, 0.f};
  // this lane's A and A^2 summed in double-float (the fp32 pipe), added to
  // the fp64 accumulators once per environment
  df a1 = zero, a2 = zero;
  df carry = zero;  // A at the step after the current chunk
  for (int64_t te = T; te > 0; te -= 32 * kJ) {
    const int64_t ts = te - 32 * kJ > 0 ? te - 32 * kJ : 0;
    df del[kJ], cc[kJ];
    df a = one, b = zero;  // this lane's steps composed: x -> b + a x
    // every input of the lane's steps is loaded before any is used, so
    // the loads share one round trip
    float rr[kJ], vv[kJ], vn[kJ];
    bool dd[kJ];
#pragma unroll
    for (int i = 0; i < kJ; ++i) {
      const int64_t t = ts + (int64_t)lane * kJ + i;
      const uint64_t at = (uint64_t)(t < te ? t : ts) * E + e;
      rr[i] = r[at];
      vv[i] = v[at];
      vn[i] = v[at + E];
      dd[i] = d[at] != 0;
    }
#pragma unroll
    for (int i = kJ - 1; i >= 0; --i) {
      const int64_t t = ts + (int64_t)lane * kJ + i;
      if (t < te) {
        const bool dn = dd[i];
        // delta = r + gamma V' (1 - d) - V
        df x = dn ? df{rr[i], 0.f} : df_add_f(df_mul_f(g, vn[i]), rr[i]);
        del[i] = df_add_f(x, -vv[i]);
        cc[i] = dn ? zero : gl;
        b = df_add(del[i], df_mul(cc[i], b));
        a = df_mul(cc[i], a);
      } else {
        del[i] = zero;
        cc[i] = one;
      }
    }
    // inclusive suffix scan: lane l gets lanes l..31 composed
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const df a2 = df_shfl_down(a, o);
      const df b2 = df_shfl_down(b, o);
      if (lane + o < 32) {
        b = df_add(b, df_mul(a, b2));
        a = df_mul(a, a2);
      }
    }
    const df an = df_shfl_down(a, 1);
    const df bn = df_shfl_down(b, 1);
    df A = lane < 31 ? df_add(bn, df_mul(an, carry)) : carry;  // A after my steps
#pragma unroll
    for (int i = kJ - 1; i >= 0; --i) {
      const int64_t t = ts + (int64_t)lane * kJ + i;
      if (t < te) {
        A = df_add(del[i], df_mul(cc[i], A));
        const uint64_t at = (uint64_t)t * E + e;
        if (A_out) A_out[at] = A.hi;
        if (ret) ret[at] = df_add_f(A, vv[i]).hi;
        a1 = df_add(a1, A);
        a2 = df_add(a2, df_mul(A, A));
      }
    }
    const df c0 = df_add(b, df_mul(a, carry));
    carry = {__shfl_sync(kFull, c0.hi, 0), __shfl_sync(kFull, c0.lo, 0)};
  }
  s1 += df_to_d(a1);
  s2 += df_to_d(a2);
}

__global__ void __launch_bounds__(kGaeThreads)
k_gae_scan(const float *__restrict__ r, const float *__restrict__ v,
           const uint8_t *__restrict__ d, uint32_t T, uint32_t E, double gamma,
           double lambda, float *__restrict__ A_out, float *__restrict__ ret,
           double *__restrict__ partial) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  pdl_wait();
  const df g = df_split(gamma);
  const df gl = df_split(gamma * lambda);
  double s1 = 0.0, s2 = 0.0;
  for (uint32_t e = blockIdx.x * kGaeWarps + wid; e < E; e += gridDim.x * kGaeWarps)
    gae_env(r, v, d, T, E, e, g, gl, A_out, ret, s1, s2);
  pdl_launch();
  if (!partial) return;  // no normalisation requested
  // per-CTA partial sums (fixed order: warps, then lanes by xor tree)
  __shared__ double ws1[kGaeWarps], ws2[kGaeWarps];
#pragma unroll
  for (int o = 16; o; o >>= 1) {
    s1 += __shfl_xor_sync(kFull, s1, o);
    s2 += __shfl_xor_sync(kFull, s2, o);
  }
  if (lane == 0) {
    ws1[wid] = s1;
    ws2[wid] = s2;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    double t1 = 0.0, t2 = 0.0;
    for (int w = 0; w < kGaeWarps; ++w) {
      t1 += ws1[w];
      t2 += ws2[w];
    }
    partial[2 * blockIdx.x] = t1;
    partial[2 * blockIdx.x + 1] = t2;
  }
}

// Sum of the per-CTA partials (sum A, sum A^2) in a fixed order: strided
// per-thread sums, then a shared-memory tree; the totals end in r1[0],
// r2[0].  Every CTA that calls it gets the same bits.
__device__ __forceinline__ void reduce_partials(const double *partial, uint32_t nparts,
                                                double *r1, double *r2) {
  double t1 = 0.0, t2 = 0.0;
  for (unsigned i = threadIdx.x; i < nparts; i += kNormThreads) {
    t1 += __ldcg(&partial[2 * i]);
    t2 += __ldcg(&partial[2 * i + 1]);
  }
  r1[threadIdx.x] = t1;
  r2[threadIdx.x] = t2;
  __syncthreads();
  for (int w = kNormThreads / 2; w > 0; w >>= 1) {
    if ((int)threadIdx.x < w) {
      r1[threadIdx.x] += r1[threadIdx.x + w];
      r2[threadIdx.x] += r2[threadIdx.x + w];
    }
    __syncthreads();
  }
}

// This rank's statistics of A for a normalisation over several ranks:
// stats = (n, sum A, sum A^2), reduced from the scan's partials in the same
// order as k_gae_norm reduces them (one CTA).
__global__ void __launch_bounds__(kNormThreads)
k_gae_stats(const double *partial, uint32_t nparts, uint64_t n, double *stats) {
  __shared__ double r1[kNormThreads], r2[kNormThreads];
  pdl_wait();
  pdl_launch();
  reduce_partials(partial, nparts, r1, r2);
  if (threadIdx.x == 0) {
    stats[0] = (double)n;
    stats[1] = r1[0];
    stats[2] = r2[0];
  }
}

// Normalisation: every CTA reduces the per-CTA partials of the scan in the
// same fixed order (or reads the statistics (n, sum A, sum A^2) of all ranks
// when `stats` is given), then one thread per element writes
// (A - mean) * inv_std.  A is read from A_src (the caller's adv, or adv_norm
// itself); n is the number of elements here.
__global__ void __launch_bounds__(kNormThreads)
k_gae_norm(const float *A_src, float *adv_norm, uint64_t n, const double *partial,
           uint32_t nparts, const double *stats) {
  __shared__ double r1[kNormThreads], r2[kNormThreads];
  __shared__ double stat[2];
  pdl_wait();
  pdl_launch();
  // this thread's first element, loaded beside the partial sums
  const uint64_t i0 = blockIdx.x * (uint64_t)kNormThreads + threadIdx.x;
  const float a0 = i0 < n ? __ldcg(&A_src[i0]) : 0.f;
  double nn = (double)n, s1, s2;
  if (stats) {
    nn = __ldcg(&stats[0]);
    s1 = __ldcg(&stats[1]);
    s2 = __ldcg(&stats[2]);
  } else {
    reduce_partials(partial, nparts, r1, r2);
    s1 = r1[0];
    s2 = r2[0];
  }
  if (threadIdx.x == 0) {
    const double mean = s1 / nn;
    double var = nn > 1.0 ? (s2 - s1 * mean) / (nn - 1.0) : 0.0;
    if (var < 0.0) var = 0.0;
    stat[0] = mean;
    // a single value equals its mean and normalises to exactly 0; the scale
    // is 0 so that the fp32 rounding of the stored A (A - mean ~ 2^-24 |A|
    // here) is not multiplied by 1 / 1e-8
    stat[1] = nn > 1.0 ? 1.0 / (sqrt(var) + 1e-8) : 0.0;
  }
  __syncthreads();
  const double mean = stat[0], inv = stat[1];
  if (i0 < n) adv_norm[i0] = (float)(((double)a0 - mean) * inv);
  for (uint64_t i = i0 + (uint64_t)gridDim.x * kNormThreads; i < n;
       i += (uint64_t)gridDim.x * kNormThreads)
    adv_norm[i] = (float)(((double)__ldcg(&A_src[i]) - mean) * inv);
}

}  // namespace

cudaError_t launch_gae(edp_ctx *c, const float *r, const float *v,
                       const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                       double lambda, float *adv, float *ret, float *adv_norm,
                       cudaStream_t s) {
  const uint64_t grid = (E + kGaeWarps - 1) / kGaeWarps;
  double *partial = nullptr;
  if (adv_norm) {
    void *blk = nullptr;
    const cudaError_t e = ctx_scratch(c, grid * 2 * sizeof(double), s, &blk);
    if (e != cudaSuccess) return e;
    partial = (double *)blk;
  }
  // A is kept between the kernels in adv, or in adv_norm itself (fp32; the
  // normalisation error this adds is below 2^-24 |A| / std)
  float *A_out = adv ? adv : adv_norm;
  cudaError_t e = launch_pdl(k_gae_scan, dim3((unsigned)grid), dim3(kGaeThreads), s,
                             r, v, d, T, E, gamma, lambda, A_out, ret, partial);
  if (e != cudaSuccess || !adv_norm) return e;
  const uint64_t n = (uint64_t)T * E;
  uint64_t ng = (n + kNormThreads - 1) / kNormThreads;
  if (ng > 4ull * c->coop_sms) ng = 4ull * c->coop_sms;
  return launch_pdl(k_gae_norm, dim3((unsigned)ng), dim3(kNormThreads), s,
                    (const float *)A_out, adv_norm, n, (const double *)partial,
                    (uint32_t)grid, (const double *)nullptr);
}

cudaError_t launch_gae_stats(edp_ctx *c, const float *r, const float *v,
                             const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                             double lambda, float *adv, float *ret, double *stats,
                             cudaStream_t s) {
  const uint64_t grid = (E + kGaeWarps - 1) / kGaeWarps;
  void *blk = nullptr;
  cudaError_t e = ctx_scratch(c, grid * 2 * sizeof(double), s, &blk);
  if (e != cudaSuccess) return e;
  double *partial = (double *)blk;
  e = launch_pdl(k_gae_scan, dim3((unsigned)grid), dim3(kGaeThreads), s, r, v, d, T, E,
                 gamma, lambda, adv, ret, partial);
  if (e != cudaSuccess) return e;
  return launch_pdl(k_gae_stats, dim3(1), dim3(kNormThreads), s, (const double *)partial,
                    (uint32_t)grid, (uint64_t)T * E, stats);
}

cudaError_t launch_gae_normalize(edp_ctx *c, const float *adv, uint64_t n,
                                 const double *stats, float *adv_norm, cudaStream_t s) {
  uint64_t ng = (n + kNormThreads - 1) / kNormThreads;
  if (ng > 4ull * c->coop_sms) ng = 4ull * c->coop_sms;
  return launch_pdl(k_gae_norm, dim3((unsigned)ng), dim3(kNormThreads), s, adv, adv_norm, n,
                    (const double *)nullptr, 0u, stats);
}

}  // namespace edp
