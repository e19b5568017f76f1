// k_gae.cu -- generalized advantage estimation with global advantage
// normalisation (Schulman et al., ICLR'16; the "computing returns/advantages"
// and "normalization" steps of on-policy ingestion, Sec. 2.2).
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
// All arithmetic is fp64; outputs are rounded once to fp32.
//
// One cooperative launch: phase 1 computes A and returns and per-CTA fp64
// sums of A and A^2; a bounded grid barrier; phase 2 forms mean and the
// unbiased standard deviation (every CTA reduces the partials in the same
// fixed order, so all agree bit for bit) and writes the normalised values.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kJ = 4;          // steps per lane per chunk
constexpr int kGaeWarps = 4;   // environments per CTA
constexpr int kGaeThreads = kGaeWarps * 32;

__global__ void __launch_bounds__(kGaeThreads)
k_gae(const float *__restrict__ r, const float *__restrict__ v,
      const uint8_t *__restrict__ d, uint32_t T, uint32_t E, double gamma,
      double lambda, float *__restrict__ adv, float *__restrict__ ret,
      float *__restrict__ adv_norm, double *__restrict__ partial, Ctrl *ctrl) {
  const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
  const double gl = gamma * lambda;
  // where A is kept between the phases (fp32; the normalisation error this
  // adds is below 2^-24 |A| / std)
  float *A_out = adv ? adv : adv_norm;
  double s1 = 0.0, s2 = 0.0;
  for (uint32_t e = blockIdx.x * kGaeWarps + wid; e < E; e += gridDim.x * kGaeWarps) {
    double carry = 0.0;  // A at the step after the current chunk
    for (int64_t te = T; te > 0; te -= 32 * kJ) {
      const int64_t ts = te - 32 * kJ > 0 ? te - 32 * kJ : 0;
      double del[kJ], cc[kJ];
      double a = 1.0, b = 0.0;  // this lane's steps composed
#pragma unroll
      for (int i = kJ - 1; i >= 0; --i) {
        const int64_t t = ts + (int64_t)lane * kJ + i;
        if (t < te) {
          const uint64_t at = (uint64_t)t * E + e;
          const double nd = d[at] ? 0.0 : 1.0;
          del[i] = (double)r[at] + gamma * (double)v[at + E] * nd - (double)v[at];
          cc[i] = gl * nd;
          b = del[i] + cc[i] * b;
          a = cc[i] * a;
        } else {
          del[i] = 0.0;
          cc[i] = 1.0;
        }
      }
      // inclusive suffix scan: lane l gets lanes l..31 composed
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const double a2 = __shfl_down_sync(kFull, a, o);
        const double b2 = __shfl_down_sync(kFull, b, o);
        if (lane + o < 32) {
          b = b + a * b2;
          a = a * a2;
        }
      }
      const double an = __shfl_down_sync(kFull, a, 1);
      const double bn = __shfl_down_sync(kFull, b, 1);
      double A = lane < 31 ? bn + an * carry : carry;  // A after my steps
#pragma unroll
      for (int i = kJ - 1; i >= 0; --i) {
        const int64_t t = ts + (int64_t)lane * kJ + i;
        if (t < te) {
          A = del[i] + cc[i] * A;
          const uint64_t at = (uint64_t)t * E + e;
          if (A_out) A_out[at] = (float)A;
          if (ret) ret[at] = (float)(A + (double)v[at]);
          s1 += A;
          s2 += A * A;
        }
      }
      carry = __shfl_sync(kFull, b + a * carry, 0);
    }
  }
  if (!adv_norm) return;  // no normalisation requested: no barrier needed
  // per-CTA partial sums (fixed order: warps, then lanes by xor tree)
  __shared__ double ws1[kGaeWarps], ws2[kGaeWarps];
  __shared__ double stat[2];
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
  grid_barrier(ctrl, gridDim.x);
  if (threadIdx.x == 0) {
    double t1 = 0.0, t2 = 0.0;
    for (unsigned bI = 0; bI < gridDim.x; ++bI) {
      t1 += *((volatile double *)&partial[2 * bI]);
      t2 += *((volatile double *)&partial[2 * bI + 1]);
    }
    const double n = (double)T * (double)E;
    const double mean = t1 / n;
    double var = (t2 - t1 * mean) / (n - 1.0);
    if (var < 0.0) var = 0.0;
    stat[0] = mean;
    stat[1] = 1.0 / (sqrt(var) + 1e-8);
  }
  __syncthreads();
  const double mean = stat[0], inv = stat[1];
  for (uint32_t e = blockIdx.x * kGaeWarps + wid; e < E; e += gridDim.x * kGaeWarps)
    for (uint32_t t = lane; t < T; t += 32) {
      const uint64_t at = (uint64_t)t * E + e;
      adv_norm[at] = (float)(((double)A_out[at] - mean) * inv);
    }
}

}  // namespace

cudaError_t launch_gae(edp_ctx *c, const float *r, const float *v,
                       const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                       double lambda, float *adv, float *ret, float *adv_norm,
                       cudaStream_t s) {
  int per_sm = 0;
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_gae, kGaeThreads, 0);
  uint64_t grid = (E + kGaeWarps - 1) / kGaeWarps;
  const uint64_t cap = (uint64_t)per_sm * c->coop_sms;
  if (grid > cap) grid = cap;
  if (grid == 0) grid = 1;
  double *partial = (double *)ctx_scratch(c, grid * 2 * sizeof(double));
  if (!partial) return cudaErrorMemoryAllocation;
  unsigned g = (unsigned)grid;
  void *args[] = {(void *)&r, (void *)&v, (void *)&d, &T, &E, &gamma, &lambda,
                  &adv, &ret, &adv_norm, &partial, &c->ctrl};
  return cudaLaunchCooperativeKernel((const void *)k_gae, dim3(g),
                                     dim3(kGaeThreads), args, 0, s);
}

}  // namespace edp
