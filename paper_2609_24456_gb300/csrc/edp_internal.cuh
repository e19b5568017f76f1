// edp_internal.cuh -- context layout, device helpers and kernel launchers
// shared by the translation units of libedp.  Not part of the ABI.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <string>

#include <nvtx3/nvToolsExt.h>

#include "edp.h"

namespace edp {

// Device-side fault flags (edp_ctrl::err).  Kernels never trap: they record a
// flag, zero the affected outputs and return; edp_sync reports the flags.
enum : uint32_t {
  DEVERR_INDEX = 1u,    // a slot index outside the sampleable range
  DEVERR_EMPTY = 2u,    // total priority 0 at sampling time
  DEVERR_TIMEOUT = 4u,  // a bounded device-side wait expired (staged delivery)
  DEVERR_TREE = 8u,     // a tree descent found no child holding its target
  DEVERR_OVERFLOW = 16u,  // packed output larger than its buffer (clipped)
};

// Small device-resident control block (one per context).
struct Ctrl {
  uint32_t err;
  uint32_t pending_q;  // deferred priority of the newest transition
  uint32_t max_q;      // running maximum priority
  uint32_t pad0[2];
  uint32_t upd_count;  // priority update: CTAs done with phase 1
  uint32_t pack_ticket;  // packed delivery: length CTAs done (calls are ordered)
  uint32_t pad;
  unsigned long long bad_index;  // first offending index (diagnostics)
  unsigned long long host_bytes;  // two-tier deliveries: bytes read from the host tier
};

constexpr int kFanout = 32;
constexpr int kMaxDepth = 7;  // 32^7 > 2^32 leaves

}  // namespace edp

struct edp_ctx {
  edp_config cfg;
  edp_storage st;  // payload and metadata pointers, device-accessible
  uint64_t cap = 0, cap_h = 0, cap_c = 0;
  uint64_t obs_bytes = 0, tok_bytes = 0;
  uint64_t total = 0;
  int defer = 0;  // next_obs: newest transition not sampleable
  // priority sum-tree: level d < depth holds 32^d uint64 sums; leaves uint32
  uint32_t depth = 0;
  uint64_t nleaves = 0;
  uint32_t *leaves = nullptr;
  uint64_t *level[edp::kMaxDepth] = {};
  void *tree_mem = nullptr;
  size_t tree_bytes = 0;  // internal sums and leaves, one block
  edp::Ctrl *ctrl = nullptr;
  // lazily grown scratch (shuffle, GAE partials)
  void *scratch = nullptr;
  size_t scratch_bytes = 0;
  void *perm_scratch = nullptr;
  size_t perm_bytes = 0;
  // priorities computed from TD errors before they are applied
  uint32_t *qbuf = nullptr;
  size_t qbuf_n = 0;
  // byte -> fl32(b/255) constants: x*R1 + x*R2 with one rounding
  float r1 = 0.f, r2 = 0.f;
  // per-channel normalisation: t = x - mean; y = t*S1 + t*S2 (one rounding)
  float nmean[4] = {}, ns1[4] = {}, ns2[4] = {}, nstd[4] = {};
  int norm_fast = 1;  // 0: the constants do not reproduce t/std -> divide
  // one-FMA normalisation bf16(fma(b, A, B)), where it reproduces the chain
  float naff_a[4] = {}, naff_b[4] = {};
  int norm_affine = 0;
  int coop_sms = 0;
  edp_counters cnt{};  // host-side traffic counters (edp_get_counters)
  uint64_t host_bytes_base = 0;  // the device's host-tier byte count at the last reset
  std::string err;
};

namespace edp {

// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------

// Philox4x32-10 (Salmon et al., SC'11).
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0,
                                               uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo0 = 0xD2511F53u * c.x;
    const uint32_t hi1 = __umulhi(0xCD9E8D57u, c.z);
    const uint32_t lo1 = 0xCD9E8D57u * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// Draw j of (seed, round, stream): counter (j, round.lo, stream, round.hi),
// key (seed.lo, seed.hi), value (word1 << 32) | word0.
__device__ __forceinline__ uint64_t philox_u64(uint64_t seed, uint32_t j,
                                               uint64_t round,
                                               uint32_t stream) {
  const uint4 o = philox4x32_10(
      make_uint4(j, (uint32_t)round, stream, (uint32_t)(round >> 32)),
      (uint32_t)seed, (uint32_t)(seed >> 32));
  return ((uint64_t)o.y << 32) | (uint64_t)o.x;
}

__device__ __forceinline__ uint64_t mulhi64(uint64_t a, uint64_t n) {
  return __umul64hi(a, n);
}

// Target of stratum k of B over a total S (stratified proportional
// sampling): the stratum is [lo, hi) = [floor(kS/B), floor((k+1)S/B)),
// computed as floor(kS/B) = ak + floor(bk/B) with S = aB + b (every term
// below 2^64), and t = lo + mulhi64(u, hi - lo) with u the Philox draw k of
// (seed, round, stream 1).  Targets never decrease with k.
__device__ __forceinline__ uint64_t stratum_target(uint64_t S, uint32_t B, uint32_t k,
                                                   uint64_t seed, uint64_t round) {
  const uint64_t a = S / B, b = S % B;
  const uint64_t lo = a * k + (b * k) / B;
  const uint64_t hi = a * (k + 1) + (b * (k + 1)) / B;
  const uint64_t u = philox_u64(seed, k, round, 1);
  return lo + mulhi64(u, hi - lo);
}

// fl32(b/255) for an integer-valued x = b in [0, 255]: r1 + r2 is 1/255 to
// ~2^-48 relative, and b/255 never lies that close to a rounding boundary
// of binary32, so one fused multiply-add rounds to the correctly rounded
// quotient.  (The host checks all 256 inputs at context creation.)
__device__ __forceinline__ float unit_f32(float x, float r1, float r2) {
  return __fmaf_rn(x, r1, __fmul_rn(x, r2));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t *>(&v);
}

// x^a for x in [2^-1000, 2^1000], fp64, written for GB300's narrow fp64
// pipe (a dependent fp64 FMA costs ~64 cycles and a divide ~500, so a
// general pow is ~6,000 cycles):
//   x = 2^e m with m in [sqrt(1/2), sqrt(2));
//   ln m = 2 atanh(s) = 2 (s + s^3/3 + s^5/5 + ...),  s = (m-1)/(m+1),
//     |s| <= 0.1716; the reciprocal 1/(m+1) is an fp32 seed refined by
//     two Newton steps (2^-23 -> 2^-92);
//   t = a (e ln 2 + ln m);  e^t = 2^n e^r,  n = rint(t / ln 2),
//     r = t - n ln 2 (ln 2 split in a high and a low part), |r| <= 0.35,
//     e^r by its Taylor polynomial.
// (Series: Abramowitz & Stegun 4.1.27 and 4.2.1.)  FULL: 11 + 17 terms,
// relative error ~1e-15; otherwise 7 + 11 terms, ~1e-10, ample for a result
// rounded to fp32.
template <bool FULL>
__device__ __forceinline__ double pow_pos(double x, double a) {
  long long bits = __double_as_longlong(x);
  int e = (int)((bits >> 52) & 0x7ff) - 1023;
  double m = __longlong_as_double((bits & 0x000fffffffffffffll) | 0x3ff0000000000000ll);
  if (m > 1.4142135623730951) {
    m *= 0.5;
    e += 1;
  }
  const double den = m + 1.0;
  double y = (double)(1.0f / (float)den);
  y = fma(y, fma(-den, y, 1.0), y);
  y = fma(y, fma(-den, y, 1.0), y);
  const double s = (m - 1.0) * y;
  const double s2 = s * s;
  double p;
  if (FULL) {
    p = 1.0 / 23;
    p = fma(p, s2, 1.0 / 21);
    p = fma(p, s2, 1.0 / 19);
    p = fma(p, s2, 1.0 / 17);
    p = fma(p, s2, 1.0 / 15);
  } else {
    p = 1.0 / 15;
  }
  p = fma(p, s2, 1.0 / 13);
  p = fma(p, s2, 1.0 / 11);
  p = fma(p, s2, 1.0 / 9);
  p = fma(p, s2, 1.0 / 7);
  p = fma(p, s2, 1.0 / 5);
  p = fma(p, s2, 1.0 / 3);
  p = fma(p, s2, 1.0);
  const double ln2_hi = 6.93147180369123816490e-01;  // 2^-32 accurate
  const double ln2_lo = 1.90821492927058770002e-10;
  const double lnm = 2.0 * s * p;
  const double t_hi = a * (double)e * ln2_hi;
  const double t_lo = a * ((double)e * ln2_lo + lnm);
  const double t = t_hi + t_lo;
  const double n = rint(t * 1.44269504088896340736);
  const double r = (t_hi - n * ln2_hi) + (t_lo - n * ln2_lo);
  double q;
  if (FULL) {
    q = 1.0 / 355687428096000.0;  // 1/17!
    q = fma(q, r, 1.0 / 20922789888000.0);
    q = fma(q, r, 1.0 / 1307674368000.0);
    q = fma(q, r, 1.0 / 87178291200.0);
    q = fma(q, r, 1.0 / 6227020800.0);
    q = fma(q, r, 1.0 / 479001600.0);
    q = fma(q, r, 1.0 / 39916800.0);
  } else {
    q = 1.0 / 39916800.0;  // 1/11!
  }
  q = fma(q, r, 1.0 / 3628800.0);
  q = fma(q, r, 1.0 / 362880.0);
  q = fma(q, r, 1.0 / 40320.0);
  q = fma(q, r, 1.0 / 5040.0);
  q = fma(q, r, 1.0 / 720.0);
  q = fma(q, r, 1.0 / 120.0);
  q = fma(q, r, 1.0 / 24.0);
  q = fma(q, r, 1.0 / 6.0);
  q = fma(q, r, 0.5);
  q = fma(q, r, 1.0);
  q = fma(q, r, 1.0);
  const long long ni = (long long)n;
  return q * __longlong_as_double((ni + 1023) << 52);
}

// Double-float arithmetic: a value is an unevaluated sum hi + lo of two
// fp32 numbers (about 48 significant bits), with Knuth's TwoSum, Dekker's
// product via FMA and the renormalisations of Hida, Li and Bailey.  Every
// operation is one IEEE rounding: the intrinsics are never contracted or
// reassociated by the compiler.
struct df {
  float hi, lo;
};
__device__ __forceinline__ df two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return {s, e};
}
__device__ __forceinline__ df quick_two_sum(float a, float b) {  // |a| >= |b|
  const float s = __fadd_rn(a, b);
  return {s, __fsub_rn(b, __fsub_rn(s, a))};
}
__device__ __forceinline__ df df_add(df a, df b) {
  df s = two_sum(a.hi, b.hi);
  const df t = two_sum(a.lo, b.lo);
  s.lo = __fadd_rn(s.lo, t.hi);
  s = quick_two_sum(s.hi, s.lo);
  s.lo = __fadd_rn(s.lo, t.lo);
  return quick_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ df df_add_f(df a, float b) {
  df s = two_sum(a.hi, b);
  s.lo = __fadd_rn(s.lo, a.lo);
  return quick_two_sum(s.hi, s.lo);
}
__device__ __forceinline__ df df_mul(df a, df b) {
  const float p = __fmul_rn(a.hi, b.hi);
  float e = __fmaf_rn(a.hi, b.hi, -p);
  e = __fmaf_rn(a.hi, b.lo, e);
  e = __fmaf_rn(a.lo, b.hi, e);
  return quick_two_sum(p, e);
}
__device__ __forceinline__ df df_mul_f(df a, float b) {
  const float p = __fmul_rn(a.hi, b);
  float e = __fmaf_rn(a.hi, b, -p);
  e = __fmaf_rn(a.lo, b, e);
  return quick_two_sum(p, e);
}
__device__ __forceinline__ df df_split(double x) {
  const float hi = (float)x;
  return {hi, (float)(x - (double)hi)};
}
__device__ __forceinline__ double df_to_d(df a) {
  return (double)a.hi + (double)a.lo;
}

// Importance weight (q_min / q_k)^beta in fp64, one rounding to fp32 (PER:
// (N P(i))^-beta over its batch maximum, in which N and the total cancel).
__device__ __forceinline__ float is_weight(uint32_t m, uint32_t qk, double beta) {
  if (qk == m) return 1.f;
  if (!qk) return 0.f;
  // m / qk with an fp32 seed and two Newton steps (no fp64 divide)
  const double d = (double)qk;
  double y = (double)(1.0f / (float)qk);
  y = fma(y, fma(-d, y, 1.0), y);
  y = fma(y, fma(-d, y, 1.0), y);
  return (float)pow_pos<false>((double)m * y, beta);
}

// L2 residency hints: payload streams through (an evict_first policy) so
// the small, reused priority tree stays resident (evict_last).
__device__ __forceinline__ uint64_t policy_stream() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t policy_keep() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t ld_keep(const uint64_t *p, uint64_t pol) {
  uint64_t v;
  asm volatile("ld.global.L2::cache_hint.u64 %0, [%1], %2;"
               : "=l"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ uint32_t ld_keep(const uint32_t *p, uint64_t pol) {
  uint32_t v;
  asm volatile("ld.global.L2::cache_hint.u32 %0, [%1], %2;"
               : "=r"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ uint32_t ld_stream(const uint32_t *p, uint64_t pol) {
  uint32_t v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.u32 %0, [%1], %2;"
               : "=r"(v) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ uint2 ld_stream(const uint2 *p, uint64_t pol) {
  uint2 v;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v2.u32 {%0, %1}, [%2], %3;"
               : "=r"(v.x), "=r"(v.y) : "l"(p), "l"(pol));
  return v;
}
__device__ __forceinline__ void st_stream(float4 *p, float4 v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.f32 [%0], {%1, %2, %3, %4}, %5;"
               :: "l"(p), "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "l"(pol)
               : "memory");
}
__device__ __forceinline__ void st_stream(uint4 *p, uint4 v, uint64_t pol) {
  asm volatile("st.global.L1::no_allocate.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;"
               :: "l"(p), "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "l"(pol)
               : "memory");
}

// ---------------------------------------------------------------------------
// Shared-memory staging: mbarriers and bulk asynchronous copies (sm_90+).
// A bulk copy global -> shared moves a contiguous run of bytes (both
// addresses 16-byte aligned, size a multiple of 16) on the copy engine of
// the SM and signals its completion on an mbarrier as a transaction count.
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_addr(const void *p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(unsigned long long *bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" :: "r"(smem_addr(bar)), "r"(count)
               : "memory");
}
// Makes initialised mbarriers visible to the async proxy (the bulk copies)
// and to the other threads once followed by a CTA barrier.
__device__ __forceinline__ void mbar_init_fence() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive(unsigned long long *bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" :: "r"(smem_addr(bar)) : "memory");
}
__device__ __forceinline__ void mbar_arrive_tx(unsigned long long *bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;"
               :: "r"(smem_addr(bar)), "r"(bytes) : "memory");
}
// Raises the bytes the current phase of `bar` waits for, without arriving.
__device__ __forceinline__ void mbar_expect_tx(unsigned long long *bar, uint32_t bytes) {
  asm volatile("mbarrier.expect_tx.relaxed.cta.shared::cta.b64 [%0], %1;"
               :: "r"(smem_addr(bar)), "r"(bytes) : "memory");
}
__device__ __forceinline__ bool mbar_test(unsigned long long *bar, uint32_t parity) {
  uint32_t ok;
  asm volatile("{\n\t.reg .pred p;\n\t"
               "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
               "selp.u32 %0, 1, 0, p;\n\t}"
               : "=r"(ok) : "r"(smem_addr(bar)), "r"(parity) : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t global_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Waits for the phase of `bar` with parity `parity` to complete; gives up
// after about `limit_ns` nanoseconds (false), so that no wait can hang.
__device__ __forceinline__ bool mbar_wait(unsigned long long *bar, uint32_t parity,
                                          uint64_t limit_ns) {
  if (mbar_test(bar, parity)) return true;
  const uint64_t t0 = global_ns();
  for (;;) {
    // the timer is read once per 64 tests: reading it more often slows the
    // waiting warps measurably (a stage's consumers poll the barrier)
    for (int i = 0; i < 64; ++i)
      if (mbar_test(bar, parity)) return true;
    if (global_ns() - t0 > limit_ns) return false;
  }
}
// bytes [src, src + n) -> shared [dst, dst + n), completion counted on bar;
// `pol` is an L2 cache policy for the source.
__device__ __forceinline__ void bulk_load(void *dst, const void *src, uint32_t n,
                                          unsigned long long *bar, uint64_t pol) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint"
      " [%0], [%1], %2, [%3], %4;"
      :: "r"(smem_addr(dst)), "l"(src), "r"(n), "r"(smem_addr(bar)), "l"(pol) : "memory");
}

__device__ __forceinline__ void flag(Ctrl *c, uint32_t bits,
                                     unsigned long long detail) {
  if ((atomicOr(&c->err, bits) & bits) == 0)
    atomicCAS(&c->bad_index, 0ull, detail + 1);
}

// Programmatic dependent launch (sm_90+): a kernel launched with
// launch_pdl may be scheduled while its predecessor in the stream is still
// running; pdl_wait() blocks until the predecessor has completed and its
// writes are visible, so every such kernel calls it before touching memory
// the predecessor may write.  pdl_launch() lets the next kernel in the
// stream start launching.  Both are no-ops for a kernel launched without
// the attribute.  The samplers, small grids that a one-wave delivery grid
// follows, call pdl_launch() at their end: triggered at their start, the
// delivery's CTAs are placed while the sampler's CTAs still hold their SMs,
// and the block scheduler packs them onto the other SMs up to the occupancy
// limit (304 CTAs on 88 of the 152 SMs), leaving the rest idle for the
// whole delivery.
__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_launch() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block,
                       cudaStream_t s, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ---------------------------------------------------------------------------
// Launchers (host).  Each returns cudaGetLastError() after its launches.
// ---------------------------------------------------------------------------
// Rows of an ingest source into the ring at first, first + 1, ... (mod
// dst_cap).  wait_first: wait for the preceding kernel before touching
// memory; false only right behind a kernel of the same call that waited on
// its own predecessor (the copy then overlaps it, and waits at its end).
cudaError_t launch_copy_rows(uint8_t *dst, uint64_t dst_cap, uint64_t first,
                             const uint8_t *src, uint64_t n, uint64_t row_bytes,
                             cudaStream_t s, bool wait_first);
cudaError_t launch_ingest_meta(edp_ctx *ctx, const edp_fields *src, uint64_t n,
                               const uint32_t *q, cudaStream_t s);
cudaError_t launch_demote(edp_ctx *ctx, uint64_t first_id, uint64_t n,
                          cudaStream_t s);
// Demotion and insertion fused, for the steady state of a full two-tier
// ring: ids first_id + j leave HBM slot (first_id + j) mod cap_h for host
// slot (first_id + j) mod cap_c while source rows j of the ingest (obs,
// tokens) take their HBM slot.
cudaError_t launch_swap(edp_ctx *ctx, uint64_t first_id, const uint8_t *obs,
                        const int32_t *tokens, uint64_t n, cudaStream_t s);
// payload, metadata and leaves of src ids [L0, L0 + n) into dst's placement
// as dst ids 0 .. n-1 (dst then has n insertions)
cudaError_t launch_migrate(const edp_ctx *src, edp_ctx *dst, uint64_t L0, uint64_t n,
                           cudaStream_t s);
// rows [src_row, src_row + n) of an ingest source -> host-tier slots of ids
// first_id .. first_id + n - 1
cudaError_t launch_copy_rows_to_host(edp_ctx *ctx, const uint8_t *obs,
                                     const int32_t *tokens, uint64_t src_row,
                                     uint64_t first_id, uint64_t n,
                                     cudaStream_t s);
// Delivery.  With `draw`, the batch is drawn by the uniform sampler inside
// the delivery kernel (idx unused; draw->idx_out receives the indices).
struct DrawUniform {
  uint64_t seed, round;
  int64_t *idx_out;
};
cudaError_t launch_deliver(edp_ctx *ctx, const int64_t *idx, uint32_t B,
                           const edp_batch *out, cudaStream_t s,
                           const DrawUniform *draw = nullptr);
// LLM post-training: group-relative advantages and packed delivery
cudaError_t launch_grpo(edp_ctx *ctx, const float *r, const uint64_t *goff, uint32_t ng,
                        float eps, float *adv, cudaStream_t s);
cudaError_t launch_pack(edp_ctx *ctx, const int32_t *tokens, const uint64_t *soff,
                        uint64_t nseq, const int64_t *idx, uint32_t B, const float *sv,
                        int32_t *otok, uint64_t *ooff, float *osv, uint64_t cap,
                        cudaStream_t s);
cudaError_t launch_grpo_pack(edp_ctx *ctx, const float *r, const uint64_t *goff, uint32_t ng,
                             float eps, float *adv, const int32_t *tokens,
                             const uint64_t *soff, uint64_t nseq, const int64_t *idx,
                             uint32_t B, int32_t *otok, uint64_t *ooff, float *osv,
                             uint64_t cap, cudaStream_t s);
cudaError_t launch_tree_refresh(edp_ctx *ctx, uint64_t first_leaf,
                                uint64_t count, cudaStream_t s);
// Nodes of each level d that cover leaves [first, first + count) (mod the
// capacity): [a0, a0 + n0) and, on a wrap, [a1, a1 + n1).
struct TreeRanges {
  uint64_t a0[kMaxDepth], n0[kMaxDepth], a1[kMaxDepth], n1[kMaxDepth];
};
void tree_ranges(const edp_ctx *ctx, uint64_t first, uint64_t count, TreeRanges *out);
// A whole insertion in one launch (single-tier rings, n small enough):
// metadata, leaves and the refresh of the tree above leaves
// [tree_first, tree_first + tree_count) by one CTA, the payload rows by
// the others.
bool ingest_fusable(const edp_ctx *ctx, uint64_t n);
cudaError_t launch_ingest_fused(edp_ctx *ctx, const edp_fields *f, uint64_t n,
                                const uint32_t *q, uint64_t tree_first,
                                uint64_t tree_count, cudaStream_t s);
cudaError_t launch_tree_build_all(edp_ctx *ctx, cudaStream_t s);
cudaError_t launch_sample_uniform(edp_ctx *ctx, uint32_t B, uint64_t seed,
                                  uint64_t round, int64_t *idx, cudaStream_t s);
cudaError_t launch_sample_prioritized(edp_ctx *ctx, uint32_t B, uint64_t seed,
                                      uint64_t round, int64_t *idx,
                                      uint32_t *q, cudaStream_t s);
// Sharded buffer (k_tree.cu, k_shard.cu)
cudaError_t launch_sample_targets(edp_ctx *ctx, const uint64_t *targets, uint32_t n,
                                  int64_t *idx, uint32_t *q, cudaStream_t s);
cudaError_t launch_tree_total(edp_ctx *ctx, uint64_t *total, cudaStream_t s);
cudaError_t launch_route_prioritized(edp_ctx *ctx, const uint64_t *totals, uint32_t G,
                                     uint32_t B, uint32_t k0, uint32_t n, uint64_t seed,
                                     uint64_t round, uint64_t *local_t, int64_t *counts,
                                     cudaStream_t s);
cudaError_t launch_batch_qmin(edp_ctx *ctx, const uint32_t *q, uint32_t n, int64_t *qmin,
                              cudaStream_t s);
cudaError_t launch_is_weights(edp_ctx *ctx, const uint32_t *q, uint32_t n,
                              const int64_t *qmin, double beta, float *w, cudaStream_t s);
cudaError_t launch_gae_stats(edp_ctx *ctx, const float *r, const float *v,
                             const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                             double lambda, float *adv, float *ret, double *stats,
                             cudaStream_t s);
cudaError_t launch_gae_normalize(edp_ctx *ctx, const float *adv, uint64_t n,
                                 const double *stats, float *adv_norm, cudaStream_t s);
cudaError_t launch_permute(edp_ctx *ctx, uint32_t n, uint64_t seed,
                           uint64_t round, int64_t *idx, cudaStream_t s);
cudaError_t launch_update(edp_ctx *ctx, const int64_t *idx, const uint32_t *q,
                          const float *td, double alpha, double eps, uint32_t n,
                          cudaStream_t s);
cudaError_t launch_prio_from_td(const float *td, uint32_t n, double alpha,
                                double eps, uint32_t *q, cudaStream_t s);
cudaError_t launch_gae(edp_ctx *ctx, const float *r, const float *v,
                       const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                       double lambda, float *adv, float *ret, float *adv_norm,
                       cudaStream_t s);
cudaError_t launch_probe_read(const void *src, uint64_t bytes, uint64_t *fold,
                              cudaStream_t s);

// Scratch owned by the context, grown on demand.  Growing allocates, and
// first waits for the device (the old block may still be in use); neither
// is allowed while `s` is being captured into a CUDA graph, so a call that
// would grow there returns cudaErrorStreamCaptureUnsupported and changes
// nothing (the caller makes one call of its largest size before capture).
// cudaErrorMemoryAllocation when the allocator fails.
cudaError_t ctx_scratch(edp_ctx *ctx, size_t bytes, cudaStream_t s, void **out);
// shuffle scratch: its first perm_zeroed_bytes() start zeroed and are left
// zeroed by every shuffle
cudaError_t ctx_perm_scratch(edp_ctx *ctx, size_t bytes, cudaStream_t s, void **out);
size_t perm_scratch_bytes(uint32_t n);
size_t perm_zeroed_bytes();
cudaError_t ctx_qbuf(edp_ctx *ctx, size_t n, cudaStream_t s, uint32_t **out);

// ---------------------------------------------------------------------------
// Host helpers shared by the entry points
// ---------------------------------------------------------------------------

// Makes `dev` the calling thread's current device for the guard's lifetime
// and gives the thread its previous current device back afterwards, so an
// entry point never changes the device its caller selected.
class DeviceGuard {
 public:
  explicit DeviceGuard(int dev) {
    if (cudaGetDevice(&prev_) != cudaSuccess) {
      cudaGetLastError();
      prev_ = -1;
    }
    if (prev_ != dev && cudaSetDevice(dev) != cudaSuccess) {
      cudaGetLastError();
      ok_ = false;
    }
    switched_ = ok_ && prev_ >= 0 && prev_ != dev;
  }
  ~DeviceGuard() {
    if (switched_) cudaSetDevice(prev_);
  }
  bool ok() const { return ok_; }
  DeviceGuard(const DeviceGuard &) = delete;
  DeviceGuard &operator=(const DeviceGuard &) = delete;

 private:
  int prev_ = -1;
  bool ok_ = true;
  bool switched_ = false;
};

// Host-side NVTX range (domain "libedp") spanning an entry point's enqueue
// work, so a timeline tool shows each call beside the kernels it launched.
// The NVTX calls are no-ops unless a tool is attached.
class TraceRange {
 public:
  explicit TraceRange(const char *name) {
    nvtxEventAttributes_t a = {};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    nvtxDomainRangePushEx(domain(), &a);
  }
  ~TraceRange() { nvtxDomainRangePop(domain()); }
  TraceRange(const TraceRange &) = delete;
  TraceRange &operator=(const TraceRange &) = delete;

 private:
  static nvtxDomainHandle_t domain() {
    static const nvtxDomainHandle_t d = nvtxDomainCreateA("libedp");
    return d;
  }
};
#define EDP_TRACE(name) ::edp::TraceRange edp_trace_range_(name)

// Resolve a caller pointer to a device-usable address.  Device memory of the
// context's GPU passes through; page-locked host memory is translated to its
// mapped device address when allow_host; pageable or foreign memory is
// rejected (false).
bool device_view(const edp_ctx *c, const void *p, const void **out, bool allow_host);

// true for page-locked host memory (reached over the host link)
bool host_memory(const void *p);

// Record a printf-style message as the context's last error; returns s.
edp_status fail(edp_ctx *c, edp_status s, const char *fmt, ...);

// The status and message for a failed launcher: EDP_ERR_OOM when scratch
// could not be allocated, EDP_ERR_STATE when scratch would have to grow
// during stream capture, EDP_ERR_CUDA otherwise.
edp_status launch_fail(edp_ctx *c, cudaError_t e, const char *where);

// Argument and state checks shared by the priority-update entry points
// (`who` names the entry point in messages): a context with a tree; for
// n > 0, idx and one of q / td given, all device memory of the context's
// GPU; with td, alpha and eps >= 0.
edp_status update_args(edp_ctx *ctx, const char *who, const int64_t *idx,
                       const uint32_t *q, const float *td, uint32_t n, double alpha,
                       double eps);

}  // namespace edp
