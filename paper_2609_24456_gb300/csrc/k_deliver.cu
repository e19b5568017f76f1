// k_deliver.cu -- fused delivery: gather the sampled transitions, transform
// their uint8 payload into the learner layout, collate metadata, and
// compute importance weights, in one pass over the payload (the delivery
// operator of Sec. 2.2: the chosen transitions are materialised in the
// layout and batch shape the learner consumes).
//
// Work decomposition: the batch's output is a flat sequence of units (a
// 32-bit word of a frame, an 8-pixel group, an 8-byte run of a plane), cut
// into warp spans whose size is set from the work, not from the grid: a
// warp runs a few iterations of its unrolled loop per span and the grid
// holds as many CTAs as that takes (several waves), so the block scheduler
// balances the tail.  (A large frame-stack batch instead streams its frames
// through shared memory: k_deliver_stack_staged below.)  A warp walks
// its span segment by segment (a segment never crosses a frame or image),
// resolving the sample's slot, episode-boundary mask and source pointer
// once per segment.  Loads are the payload bytes a lane needs for one
// 16-byte output store, so every warp-wide store instruction writes 512
// contiguous bytes.  The byte->float step is x = b (exact),
// fl32(b/255) = fma(x, r1, x*r2) with one rounding (see unit_f32), then
// optionally the per-channel normalisation and the round-to-nearest-even
// bfloat16 conversion.  Where one FMA per byte, bf16(fma(b, A_c, B_c)),
// gives the same bf16 as that chain for all 256 bytes of every channel
// (constants searched and checked on the host at creation), the
// normalising delivery uses it instead of the five-operation chain.
//
// These kernels are HBM-bound: per sample they read the unique source bytes
// once and write the (2-8x larger) output once.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// loads in flight per lane (6 x 8 bytes) in the normalising delivery
constexpr int kNormUnroll = 6;

// unrolled rows per warp iteration and iterations per warp (chunk span) of
// each kernel
constexpr int kStackUnroll = 4;
constexpr int kStackMinBlocks = 6;  // __launch_bounds__: at most 40 registers
constexpr int kHwcUnroll = 2, kHwcIters = 2;
constexpr int kNormIters = 2;

struct Common {
  const int64_t *idx;
  uint32_t B;
  uint64_t cap, oldest, nvalid;
  const int32_t *action;
  const float *reward;
  const uint8_t *done;
  int32_t *act_out;
  float *rew_out;
  uint8_t *done_out;
  const uint32_t *q;
  float *isw;
  double beta;
  const float *gsrc0, *gsrc1;
  float *gdst0, *gdst1;
  Ctrl *ctrl;
  float r1, r2;
  // fused uniform sampling: idx is then an output, sample k is drawn here
  int draw;
  uint64_t seed, round;
  int64_t *idx_out;
};

// Resolve slot -> logical offset; false (and a flag) when not sampleable.
__device__ __forceinline__ bool sample_slot(const Common &c, uint32_t k,
                                            uint64_t *slot, uint64_t *off,
                                            bool report) {
  if (c.draw) {
    // the uniform sampler's draw (Philox stream 0), made where it is used;
    // the warp that delivers the sample's first unit writes its index
    const uint64_t o = mulhi64(philox_u64(c.seed, k, c.round, 0), c.nvalid);
    const uint64_t t = c.oldest + o;
    *slot = t >= c.cap ? t - c.cap : t;
    *off = o;
    if (report) c.idx_out[k] = (int64_t)*slot;
    return true;
  }
  const int64_t s = c.idx[k];
  if (s < 0 || (uint64_t)s >= c.cap) {
    if (report) flag(c.ctrl, DEVERR_INDEX, (unsigned long long)s);
    return false;
  }
  const uint64_t o = (uint64_t)s >= c.oldest ? (uint64_t)s - c.oldest
                                             : (uint64_t)s + c.cap - c.oldest;
  if (o >= c.nvalid) {
    if (report) flag(c.ctrl, DEVERR_INDEX, (unsigned long long)s);
    return false;
  }
  *slot = (uint64_t)s;
  *off = o;
  return true;
}

// Minimum of q over the batch (one warp): loads are issued 8 per lane at a
// time so a batch of 512 costs two memory round trips, not sixteen.
__device__ __forceinline__ uint32_t batch_qmin(const Common &c, int lane) {
  uint32_t m = 0xffffffffu;
  for (uint32_t i0 = lane; i0 < c.B; i0 += 32 * 8) {
    uint32_t v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      const uint32_t i = i0 + u * 32;
      v[u] = i < c.B ? __ldg(c.q + i) : 0xffffffffu;
    }
#pragma unroll
    for (int u = 0; u < 8; ++u) m = min(m, v[u]);
  }
#pragma unroll
  for (int o = 16; o; o >>= 1) m = min(m, __shfl_xor_sync(kFull, m, o));
  return m;
}

// Per-sample collate, importance weight and scalar gathers (one warp).  The
// head warp of each sample runs this before its payload span, so the fp64
// chain of the weight overlaps the other warps' streaming.
__device__ void collate(const Common &c, uint32_t k, bool ok, uint64_t slot,
                        uint64_t off, int lane) {
  if (lane == 0) {
    if (c.act_out) c.act_out[k] = ok ? c.action[slot] : 0;
    if (c.rew_out) c.rew_out[k] = ok ? c.reward[slot] : 0.f;
    if (c.done_out) c.done_out[k] = ok ? c.done[slot] : (uint8_t)0;
    if (c.gdst0) c.gdst0[k] = ok ? c.gsrc0[off] : 0.f;
    if (c.gdst1) c.gdst1[k] = ok ? c.gsrc1[off] : 0.f;
  }
  if (c.isw) {
    // PER: w = (q_min / q_k)^beta, q_min over the batch; fp64, one rounding
    const uint32_t m = batch_qmin(c, lane);
    if (lane == 0) c.isw[k] = is_weight(m, c.q[k], c.beta);
  }
}

// The whole batch's collate, importance weights and index reporting by one
// CTA, for a frame-stack batch small enough to run one chunk per CTA: the
// streaming CTAs then carry no collate latency (q_min over the batch once, a
// block reduction, then one sample per thread).
__device__ void collate_batch(const Common &c) {
  __shared__ uint32_t s_min[kWarps];
  const int lane = threadIdx.x & 31;
  uint32_t m = 0xffffffffu;
  if (c.isw) {
    for (uint32_t i0 = threadIdx.x; i0 < c.B; i0 += kThreads * 4) {
      uint32_t v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint32_t i = i0 + u * kThreads;
        v[u] = i < c.B ? __ldg(c.q + i) : 0xffffffffu;
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) m = min(m, v[u]);
    }
#pragma unroll
    for (int o = 16; o; o >>= 1) m = min(m, __shfl_xor_sync(kFull, m, o));
    if (lane == 0) s_min[threadIdx.x >> 5] = m;
    __syncthreads();
#pragma unroll
    for (int w = 0; w < kWarps; ++w) m = min(m, s_min[w]);
  }
  for (uint32_t k = threadIdx.x; k < c.B; k += kThreads) {
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, k, &slot, &off, true);
    if (c.act_out) c.act_out[k] = ok ? c.action[slot] : 0;
    if (c.rew_out) c.rew_out[k] = ok ? c.reward[slot] : 0.f;
    if (c.done_out) c.done_out[k] = ok ? c.done[slot] : (uint8_t)0;
    if (c.gdst0) c.gdst0[k] = ok ? c.gsrc0[off] : 0.f;
    if (c.gdst1) c.gdst1[k] = ok ? c.gsrc1[off] : 0.f;
    if (c.isw) c.isw[k] = is_weight(m, c.q[k], c.beta);
  }
}

// [*f, *end): this warp's contiguous share of `total` units, rounded up to
// whole 32-unit rows so lanes stay aligned with the rows of the output.
__device__ __forceinline__ void warp_span(uint64_t total, uint64_t *f,
                                          uint64_t *end) {
  const uint64_t nw = (uint64_t)gridDim.x * kWarps;
  const uint64_t gw = (uint64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
  const uint64_t span = (((total + nw - 1) / nw) + 31) & ~31ull;
  *f = gw * span;
  *end = min(total, *f + span);
}

// exact integer -> float for a byte: 0x4B0000bb is 2^23 + b
__device__ __forceinline__ float byte_f(uint32_t w, int i) {
  return __int_as_float(__byte_perm(w, 0x4Bu, 0x4550u | i)) - 8388608.0f;
}

// ---------------------------------------------------------------------------
// Frame stack, float32 (DQN), on the load / store units.  A unit is one
// 32-bit word of frame m in [0, U) of sample k -- the frame at logical
// offset j = off - K + 1 + m, which is obs slot m (m < K) and next_obs slot
// m - 1 (m >= 1).  A lane turns its word into one float4 and stores it to
// obs and / or next_obs, so every warp-wide store writes 512 contiguous
// bytes.  Per segment (the part of one frame inside a warp's span) the warp
// resolves the slot and the episode mask once: lanes 0..K-m-1 load the done
// flags of offsets j..off and a ballot gives "an episode end before the
// anchor" (zeroes the frame in obs and next_obs) and "at the anchor" (zeroes
// it in next_obs only).
//
// This direct form serves batches too small to fill the GPU with staged
// pieces (below): one chunk per CTA, no work counter, and one more CTA
// collates the whole batch (collate_batch) so that no streaming warp waits
// on it.
// ---------------------------------------------------------------------------
struct StackArgs {
  const uint8_t *frames;
  uint32_t F;     // bytes per frame (multiple of 16)
  uint32_t W;     // 32-bit words per frame
  uint32_t K;
  uint32_t U;     // frames per sample (K, or K + 1 with next_obs)
  uint32_t span;  // units per warp per chunk (multiple of 32)
  float *obs;
  float *next;
};

// Stack units [f, end) of one warp.
template <int UN>
__device__ __forceinline__ void stack_span(const Common &c, const StackArgs &a,
                                           uint64_t f, uint64_t end, int lane,
                                           uint64_t pol) {
  const uint64_t per = (uint64_t)a.U * a.W;  // units per sample
  const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
  while (f < end) {
    const uint32_t k = (uint32_t)(f / per);
    const uint32_t rem = (uint32_t)(f - (uint64_t)k * per);
    const uint32_t m = rem / a.W;
    const uint32_t w_lo = rem - m * a.W;
    const uint64_t seg_end = min(end, (uint64_t)k * per + (uint64_t)(m + 1) * a.W);
    const uint32_t w_hi = (uint32_t)(seg_end - (uint64_t)k * per - (uint64_t)m * a.W);
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, k, &slot, &off, false);
    const int64_t j = (int64_t)off - (int64_t)(a.K - 1) + (int64_t)m;
    const bool has_obs = m < a.K;
    const bool has_next = a.next && m >= 1;
    // the payload words of the first iteration are loaded before the
    // episode flags are known (a frame the flags zero is read for nothing),
    // so the flag and payload round trips overlap
    const bool src_ok = ok && j >= 0;
    const uint64_t js = c.oldest + (uint64_t)(j < 0 ? 0 : j);
    const uint32_t *src = reinterpret_cast<const uint32_t *>(
        a.frames + (js >= c.cap ? js - c.cap : js) * a.F);
    uint32_t v[UN];
#pragma unroll
    for (int u = 0; u < UN; ++u) {
      const uint32_t w = w_lo + lane + u * 32;
      v[u] = (src_ok && w < w_hi) ? ld_stream(src + w, pol) : 0u;
    }
    bool end_before = false, end_at = false;
    if (ok && j >= 0 && (int64_t)off >= j) {
      const uint32_t span = (uint32_t)((int64_t)off - j + 1);  // 1..K
      bool d = false;
      if ((uint32_t)lane < span) {
        const uint64_t t2 = c.oldest + (uint64_t)j + lane;
        d = c.done[t2 >= c.cap ? t2 - c.cap : t2] != 0;
      }
      const unsigned bal = __ballot_sync(kFull, d);
      end_at = (bal >> (span - 1)) & 1u;
      end_before = (bal & ((1u << (span - 1)) - 1u)) != 0;
    }
    const bool zo = !ok || j < 0 || end_before;
    const bool zn = zo || end_at;
    const bool load = (has_obs && !zo) || (has_next && !zn);
    float4 *dobs = has_obs ? reinterpret_cast<float4 *>(
                                 a.obs + ((uint64_t)k * a.K + m) * a.F)
                           : nullptr;
    float4 *dnext = has_next ? reinterpret_cast<float4 *>(
                                   a.next + ((uint64_t)k * a.K + m - 1) * a.F)
                             : nullptr;
    for (uint32_t u0 = w_lo + lane; u0 < w_hi; u0 += 32 * UN) {
      if (u0 != w_lo + lane) {
#pragma unroll
        for (int u = 0; u < UN; ++u) {
          const uint32_t w = u0 + u * 32;
          v[u] = (load && w < w_hi) ? ld_stream(src + w, pol) : 0u;
        }
      }
#pragma unroll
      for (int u = 0; u < UN; ++u) {
        const uint32_t w = u0 + u * 32;
        if (w >= w_hi) continue;
        float4 fv;
        fv.x = unit_f32(byte_f(v[u], 0), c.r1, c.r2);
        fv.y = unit_f32(byte_f(v[u], 1), c.r1, c.r2);
        fv.z = unit_f32(byte_f(v[u], 2), c.r1, c.r2);
        fv.w = unit_f32(byte_f(v[u], 3), c.r1, c.r2);
        if (dobs) st_stream(dobs + w, zo ? zero4 : fv, pol);
        if (dnext) st_stream(dnext + w, zn ? zero4 : fv, pol);
      }
    }
    f = seg_end;
  }
}

template <int UN>
__global__ void __launch_bounds__(kThreads, kStackMinBlocks)
k_deliver_stack(Common c, StackArgs a) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  if (blockIdx.x == 0) {  // CTA 0 collates the batch
    collate_batch(c);
    return;
  }
  const uint64_t total = (uint64_t)c.B * a.U * a.W;
  const uint64_t f = (uint64_t)(blockIdx.x - 1) * kWarps * a.span + (uint64_t)warp * a.span;
  if (f < total) stack_span<UN>(c, a, f, min(total, f + a.span), lane, pol);
}

// ---------------------------------------------------------------------------
// Frame stack, float32, staged through shared memory (batches that fill the
// GPU).  A unit is one piece of one frame: piece p of frame m of sample k,
// where frame m is the one at logical offset off - K + 1 + m (obs slot m for
// m < K, next_obs slot m - 1 for m >= 1), and the npieces pieces of a frame
// are equal runs of at most kPiece bytes.  Units are dealt to the CTAs round
// robin (unit u to CTA u mod grid): equal units, so the split is balanced
// without a work counter, and no state outlives the launch.  Per CTA:
//  - warp 0 (producer) resolves 32 of its units at a time, a lane each:
//    index -> slot and logical offset -> source address, and the done flags
//    of the frame's window (offsets j .. off).  It issues the bulk copy of
//    each unit's piece into a free stage as soon as the address is known,
//    before the flags have arrived (a frame they then zero everywhere is
//    copied for nothing), and publishes the unit -- which of its output
//    copies are zero -- with its arrival on the stage once they have;
//  - warp 1 collates this CTA's samples (k = blockIdx.x mod grid): action,
//    reward, done, gathered scalars, the importance weight, and the index
//    when the batch is drawn here;
//  - warps 2 .. kStageWarps + 1 (consumers) wait for the stage, turn its
//    bytes into floats and store them to obs and / or next_obs (zeros where
//    the episode mask says so; each warp-wide store writes 512 contiguous
//    bytes), then release the stage.
// A stage's phase completes when the producer has arrived and the copy's
// bytes have landed.  kStages stages keep several pieces in flight per CTA,
// so the index -> flags chain is paid once per 32 units, beside the copies.
// Every wait is bounded (kWaitNs): on expiry the warp records DEVERR_TIMEOUT
// and stops, the producer after waiting (bounded again) for the copies it
// has in flight.
// ---------------------------------------------------------------------------
constexpr int kStages = 6;
constexpr uint32_t kPiece = 7168;  // bytes per stage, a multiple of 16
constexpr int kStageWarps = 7;     // consumer warps
constexpr int kStagedThreads = 32 * (kStageWarps + 2);
constexpr int kStagedPerSm = 2;    // CTAs per SM in the grid
constexpr int kStagedUnroll = 4;
constexpr uint64_t kWaitNs = 1000000000ull;
// unit flags (StageSmem::meta)
constexpr uint32_t kZeroObs = 1u, kZeroNext = 2u, kLoaded = 4u;

struct StageSmem {
  alignas(128) uint8_t buf[kStages][kPiece];
  unsigned long long full[kStages];   // producer -> consumers (bytes landed)
  unsigned long long empty[kStages];  // consumers -> producer (stage free)
  uint32_t meta[kStages];
};

// Collate of samples first, first + stride, ... (one warp): q_min over the
// batch once, then one sample per lane.
__device__ void collate_strided(const Common &c, uint32_t first, uint32_t stride, int lane) {
  const uint32_t m = c.isw ? batch_qmin(c, lane) : 0u;
  for (uint64_t k = first + (uint64_t)lane * stride; k < c.B; k += 32ull * stride) {
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, (uint32_t)k, &slot, &off, true);
    if (c.act_out) c.act_out[k] = ok ? c.action[slot] : 0;
    if (c.rew_out) c.rew_out[k] = ok ? c.reward[slot] : 0.f;
    if (c.done_out) c.done_out[k] = ok ? c.done[slot] : (uint8_t)0;
    if (c.gdst0) c.gdst0[k] = ok ? c.gsrc0[off] : 0.f;
    if (c.gdst1) c.gdst1[k] = ok ? c.gsrc1[off] : 0.f;
    if (c.isw) c.isw[k] = is_weight(m, c.q[k], c.beta);
  }
}

// Unit u -> (sample k, frame m, piece p).
struct Unit {
  uint32_t k, m, p;
};
__device__ __forceinline__ Unit unit_of(uint64_t u, uint32_t U, uint32_t npieces) {
  const uint32_t per_k = U * npieces;
  Unit r;
  r.k = (uint32_t)(u / per_k);
  const uint32_t rem = (uint32_t)(u - (uint64_t)r.k * per_k);
  r.m = rem / npieces;
  r.p = rem - r.m * npieces;
  return r;
}

__device__ void stage_producer(const Common &c, const StackArgs &a, StageSmem &sm,
                               uint32_t npieces, uint32_t piece, uint64_t nmine,
                               int lane, uint64_t pol) {
  for (uint64_t i0 = 0; i0 < nmine; i0 += 32) {
    // lane l resolves unit i0 + l of this CTA: its source now, its episode
    // flags in flight (used when the unit is published)
    uint64_t src = 0;
    bool valid = false, ok = false, has_obs = false, has_next = false;
    int64_t span = 0;
    uint32_t bits = 0;
    if (i0 + lane < nmine) {
      valid = true;
      const Unit t = unit_of(blockIdx.x + (i0 + lane) * gridDim.x, a.U, npieces);
      uint64_t slot = 0, off = 0;
      ok = sample_slot(c, t.k, &slot, &off, false);
      const int64_t j = (int64_t)off - (int64_t)(a.K - 1) + (int64_t)t.m;
      has_obs = t.m < a.K;
      has_next = a.next && t.m >= 1;
      if (ok && j >= 0) {
        uint64_t js = c.oldest + (uint64_t)j;
        if (js >= c.cap) js -= c.cap;
        src = (uint64_t)(a.frames + js * a.F + (uint64_t)t.p * piece);
        span = (int64_t)off - j + 1;  // flags of offsets j .. off (<= K)
      } else {
        ok = false;  // zero in every copy
      }
      // bit i: done flag of offset j + i
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        if (i < span) {
          uint64_t ps = c.oldest + (uint64_t)(off - (uint64_t)(span - 1)) + i;
          if (ps >= c.cap) ps -= c.cap;
          bits |= (c.done[ps] != 0 ? 1u : 0u) << i;
        }
      }
    }
    const uint32_t n = (uint32_t)min((uint64_t)32, nmine - i0);
    uint32_t pub = 0;  // units of the group published so far
    uint32_t good = 1;
    // this lane's unit flags: an episode end before the anchor zeroes the
    // frame in obs and next_obs; one at the anchor zeroes it in next_obs
    // only (evaluated when the first unit is published: the flag loads are
    // in flight until then)
    uint32_t fl = 0;
    bool fl_ready = false;
#define EDP_PUBLISH()                                                            \
    do {                                                                         \
      if (!fl_ready) {                                                           \
        const bool end_before = span > 1 && (bits & ((1u << (span - 1)) - 1u)) != 0; \
        const bool end_at = span > 0 && ((bits >> (span - 1)) & 1u);             \
        const bool zo = !ok || end_before, zn = zo || end_at;                    \
        const bool load = (has_obs && !zo) || (has_next && !zn);                 \
        fl = valid ? (zo ? kZeroObs : 0u) | (zn ? kZeroNext : 0u) | (load ? kLoaded : 0u) \
                   : 0u;                                                         \
        fl_ready = true;                                                         \
      }                                                                          \
      const uint32_t fl_t = __shfl_sync(kFull, fl, pub);                         \
      if (lane == 0) {                                                           \
        const int st_p = (int)((i0 + pub) % kStages);                            \
        sm.meta[st_p] = fl_t;                                                    \
        mbar_arrive(&sm.full[st_p]);                                             \
      }                                                                          \
      ++pub;                                                                     \
    } while (0)
    uint32_t t = 0;
    for (; t < n; ++t) {
      const uint64_t i = i0 + t;
      const int st = (int)(i % kStages);
      if (i >= kStages) {
        // the stage's previous occupant (unit i - kStages) must have been
        // published before the consumers can free the stage
        while (pub + kStages <= t) EDP_PUBLISH();
        if (lane == 0)
          good = mbar_wait(&sm.empty[st], (uint32_t)((i / kStages) - 1) & 1u, kWaitNs);
        good = __shfl_sync(kFull, good, 0);
        if (!good) break;
      }
      const uint64_t src_t = __shfl_sync(kFull, src, t);
      if (lane == 0 && src_t) {
        mbar_expect_tx(&sm.full[st], piece);
        bulk_load(sm.buf[st], reinterpret_cast<const void *>(src_t), piece, &sm.full[st], pol);
      }
    }
    if (!good) {
      // units i0 + pub .. i0 + t - 1 are issued but unpublished: publish
      // them so their phases can complete, then wait (bounded) for the
      // bytes of the last kStages issued copies, which land in this CTA's
      // shared memory, before the CTA may exit
      while (pub < t) EDP_PUBLISH();
      if (lane == 0) {
        const uint64_t end = i0 + t;
        flag(c.ctrl, DEVERR_TIMEOUT, end);
        for (uint64_t q = end > kStages ? end - kStages : 0; q < end; ++q)
          mbar_wait(&sm.full[q % kStages], (uint32_t)(q / kStages) & 1u, kWaitNs);
      }
      return;
    }
    while (pub < n) EDP_PUBLISH();
#undef EDP_PUBLISH
  }
}

__device__ void stage_consumer(const Common &c, const StackArgs &a, StageSmem &sm,
                               uint32_t npieces, uint32_t piece, uint64_t nmine,
                               int cw, int lane, uint64_t pol) {
  const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
  const uint32_t W = piece / 4;  // words of a piece
  constexpr uint32_t kRow = 32 * kStageWarps;
  for (uint64_t i = 0; i < nmine; ++i) {
    const int st = (int)(i % kStages);
    if (!mbar_wait(&sm.full[st], (uint32_t)(i / kStages) & 1u, kWaitNs)) {
      if (lane == 0) flag(c.ctrl, DEVERR_TIMEOUT, i);
      return;
    }
    const uint32_t fl = sm.meta[st];
    const Unit t = unit_of(blockIdx.x + i * gridDim.x, a.U, npieces);
    const bool zo = fl & kZeroObs, zn = fl & kZeroNext, loaded = fl & kLoaded;
    const uint64_t pofs = (uint64_t)t.p * piece;
    float4 *dobs = t.m < a.K ? reinterpret_cast<float4 *>(
                                   a.obs + ((uint64_t)t.k * a.K + t.m) * a.F + pofs)
                             : nullptr;
    float4 *dnext = (a.next && t.m >= 1)
                        ? reinterpret_cast<float4 *>(
                              a.next + ((uint64_t)t.k * a.K + t.m - 1) * a.F + pofs)
                        : nullptr;
    const uint32_t *src = reinterpret_cast<const uint32_t *>(sm.buf[st]);
    for (uint32_t w0 = cw * 32 + lane; w0 < W; w0 += kRow * kStagedUnroll) {
      uint32_t v[kStagedUnroll];
#pragma unroll
      for (int u = 0; u < kStagedUnroll; ++u) {
        const uint32_t w = w0 + u * kRow;
        v[u] = (loaded && w < W) ? src[w] : 0u;
      }
#pragma unroll
      for (int u = 0; u < kStagedUnroll; ++u) {
        const uint32_t w = w0 + u * kRow;
        if (w >= W) continue;
        float4 fv;
        fv.x = unit_f32(byte_f(v[u], 0), c.r1, c.r2);
        fv.y = unit_f32(byte_f(v[u], 1), c.r1, c.r2);
        fv.z = unit_f32(byte_f(v[u], 2), c.r1, c.r2);
        fv.w = unit_f32(byte_f(v[u], 3), c.r1, c.r2);
        if (dobs) st_stream(dobs + w, zo ? zero4 : fv, pol);
        if (dnext) st_stream(dnext + w, zn ? zero4 : fv, pol);
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&sm.empty[st]);
  }
}

__global__ void __launch_bounds__(kStagedThreads)
k_deliver_stack_staged(Common c, StackArgs a, uint32_t npieces, uint32_t piece) {
  __shared__ StageSmem sm;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&sm.full[i], 1);
      mbar_init(&sm.empty[i], kStageWarps);
    }
    mbar_init_fence();
  }
  __syncthreads();
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  const uint64_t units = (uint64_t)c.B * a.U * npieces;
  const uint64_t nmine =
      units > blockIdx.x ? (units - blockIdx.x + gridDim.x - 1) / gridDim.x : 0;
  if (warp == 0)
    stage_producer(c, a, sm, npieces, piece, nmine, lane, pol);
  else if (warp == 1)
    collate_strided(c, blockIdx.x, gridDim.x, lane);
  else
    stage_consumer(c, a, sm, npieces, piece, nmine, warp - 2, lane, pol);
}

// ---------------------------------------------------------------------------
// HWC uint8 -> CHW bfloat16 (on-policy mini-batches).  Unit = 8 pixels: a lane
// converts 8 consecutive pixels: it loads their 8*C interleaved bytes and
// writes C 16-byte runs, one per channel plane.
// ---------------------------------------------------------------------------
struct ChwArgs {
  const uint8_t *obs;
  uint32_t HW;   // pixels per image
  __nv_bfloat16 *out;
};

template <int C, int UN>
__global__ void __launch_bounds__(kThreads)
k_deliver_hwc(Common c, ChwArgs a) {
  const int lane = threadIdx.x & 31;
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  const uint32_t G = a.HW / 8;  // 8-pixel groups per image
  const uint64_t total = (uint64_t)c.B * G;
  const uint64_t F = (uint64_t)a.HW * C;
  uint64_t f, end;
  warp_span(total, &f, &end);
  while (f < end) {
    const uint32_t k = (uint32_t)(f / G);
    const uint32_t g_lo = (uint32_t)(f - (uint64_t)k * G);
    const uint64_t seg_end = min(end, (uint64_t)(k + 1) * G);
    const uint32_t g_hi = (uint32_t)(seg_end - (uint64_t)k * G);
    const bool head = g_lo == 0;
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, k, &slot, &off, head && lane == 0);
    if (head) collate(c, k, ok, slot, off, lane);
    const uint2 *src = reinterpret_cast<const uint2 *>(a.obs + slot * F);
    uint4 *dst = reinterpret_cast<uint4 *>(a.out + (uint64_t)k * F);
    for (uint32_t g0 = g_lo + lane; g0 < g_hi; g0 += 32 * UN) {
      uint2 v[UN][C];
#pragma unroll
      for (int u = 0; u < UN; ++u) {
        const uint32_t g = g0 + u * 32;
#pragma unroll
        for (int q = 0; q < C; ++q)
          v[u][q] = (ok && g < g_hi) ? ld_stream(src + (uint64_t)g * C + q, pol)
                                     : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < UN; ++u) {
        const uint32_t g = g0 + u * 32;
        if (g >= g_hi) continue;
        uint32_t wd[2 * C];
#pragma unroll
        for (int q = 0; q < C; ++q) {
          wd[2 * q] = v[u][q].x;
          wd[2 * q + 1] = v[u][q].y;
        }
#pragma unroll
        for (int ch = 0; ch < C; ++ch) {
          float fv[8];
#pragma unroll
          for (int px = 0; px < 8; ++px) {
            const int byte = px * C + ch;  // position within the 8*C bytes
            fv[px] = unit_f32(byte_f(wd[byte >> 2], byte & 3), c.r1, c.r2);
          }
          uint4 o;
          o.x = pack_bf16x2(fv[0], fv[1]);
          o.y = pack_bf16x2(fv[2], fv[3]);
          o.z = pack_bf16x2(fv[4], fv[5]);
          o.w = pack_bf16x2(fv[6], fv[7]);
          st_stream(dst + (uint64_t)ch * G + g, o, pol);
        }
      }
    }
    f = seg_end;
  }
}

// ---------------------------------------------------------------------------
// CHW uint8 -> per-channel normalised bfloat16 (multimodal payloads), with
// token collate; optionally two-tier (payload of older transitions in
// page-locked host memory, read over the host link).  Unit = 8 bytes: a lane
// converts 8 consecutive bytes of one channel plane to one 16-byte store.
// ---------------------------------------------------------------------------
struct NormArgs {
  const uint8_t *obs_h;   // HBM ring [cap_h][F]
  const uint8_t *obs_c;   // host ring [cap_c][F] (device-mapped) or null
  const int32_t *tok_h;
  const int32_t *tok_c;
  uint64_t cap_h, cap_c, total, size;
  uint32_t F8;    // 8-byte units per image
  uint32_t HW8;   // 8-byte units per channel plane
  uint32_t L16;   // 16-byte units of tokens per transition
  float mean[4], s1[4], s2[4], sd[4];
  float aa[4], ab[4];  // one-FMA form (AFF): bf16(fma(b, aa, ab))
  int fast;
  __nv_bfloat16 *out;
  int32_t *tok_out;
};

template <int UN, bool AFF>
__global__ void __launch_bounds__(kThreads)
k_deliver_norm(Common c, NormArgs a) {
  const int lane = threadIdx.x & 31;
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  const uint64_t total = (uint64_t)c.B * a.F8;
  uint64_t f, end;
  warp_span(total, &f, &end);
  while (f < end) {
    const uint32_t k = (uint32_t)(f / a.F8);
    const uint32_t u_lo = (uint32_t)(f - (uint64_t)k * a.F8);
    const uint64_t seg_end = min(end, (uint64_t)(k + 1) * a.F8);
    const uint32_t u_hi = (uint32_t)(seg_end - (uint64_t)k * a.F8);
    const bool head = u_lo == 0;
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, k, &slot, &off, head && lane == 0);
    if (head) collate(c, k, ok, slot, off, lane);
    // tier of the logical id L = total - size + off
    const uint64_t L = a.total - a.size + off;
    const uint64_t in_hbm = a.total < a.cap_h ? a.total : a.cap_h;
    const bool hbm = !a.obs_c || L >= a.total - in_hbm;
    const uint64_t ps = hbm ? L % a.cap_h : L % a.cap_c;
    const uint8_t *obs = hbm ? a.obs_h : a.obs_c;
    const uint2 *src = reinterpret_cast<const uint2 *>(obs + ps * a.F8 * 8ull);
    uint4 *dst = reinterpret_cast<uint4 *>(a.out + (uint64_t)k * a.F8 * 8ull);
    for (uint32_t u0 = u_lo + lane; u0 < u_hi; u0 += 32 * UN) {
      uint2 v[UN];
#pragma unroll
      for (int u = 0; u < UN; ++u) {
        const uint32_t w = u0 + u * 32;
        // HBM tier: streaming non-coherent loads; host tier: plain loads of
        // the mapped page-locked memory
        v[u] = (ok && w < u_hi) ? (hbm ? ld_stream(src + w, pol) : src[w])
                                : make_uint2(0u, 0u);
      }
#pragma unroll
      for (int u = 0; u < UN; ++u) {
        const uint32_t w = u0 + u * 32;
        if (w >= u_hi) continue;
        const uint32_t ch = (w >= a.HW8) + (w >= 2 * a.HW8) + (w >= 3 * a.HW8);
        float fv[8];
        if constexpr (AFF) {
          const float A = a.aa[ch], Bc = a.ab[ch];
#pragma unroll
          for (int bb = 0; bb < 8; ++bb)
            fv[bb] = __fmaf_rn(byte_f(bb < 4 ? v[u].x : v[u].y, bb & 3), A, Bc);
        } else {
          const float mc = a.mean[ch], s1 = a.s1[ch], s2 = a.s2[ch];
#pragma unroll
          for (int bb = 0; bb < 8; ++bb) {
            const float x = unit_f32(byte_f(bb < 4 ? v[u].x : v[u].y, bb & 3), c.r1, c.r2);
            const float tt = __fsub_rn(x, mc);
            fv[bb] = a.fast ? __fmaf_rn(tt, s1, __fmul_rn(tt, s2)) : __fdiv_rn(tt, a.sd[ch]);
          }
        }
        uint4 o;
        o.x = pack_bf16x2(fv[0], fv[1]);
        o.y = pack_bf16x2(fv[2], fv[3]);
        o.z = pack_bf16x2(fv[4], fv[5]);
        o.w = pack_bf16x2(fv[6], fv[7]);
        if (!ok) o = make_uint4(0u, 0u, 0u, 0u);
        st_stream(dst + w, o, pol);
      }
    }
    if (head) {
      // a two-tier row read over the host link (edp_get_counters)
      if (lane == 0 && ok && a.obs_c && !hbm)
        atomicAdd(&c.ctrl->host_bytes,
                  (unsigned long long)a.F8 * 8ull + (a.tok_out ? a.L16 * 16ull : 0ull));
      if (a.tok_out) {
        // the row's tokens, kTokBatch 16-byte loads per lane in flight
        // before their stores
        constexpr int kTokBatch = 4;
        const uint4 *ts = reinterpret_cast<const uint4 *>(
            (hbm ? a.tok_h : a.tok_c) + ps * a.L16 * 4ull);
        uint4 *td = reinterpret_cast<uint4 *>(a.tok_out + (uint64_t)k * a.L16 * 4ull);
        for (uint32_t i0 = lane; i0 < a.L16; i0 += 32 * kTokBatch) {
          uint4 t4[kTokBatch];
#pragma unroll
          for (int u = 0; u < kTokBatch; ++u) {
            const uint32_t i = i0 + u * 32;
            t4[u] = (ok && i < a.L16) ? ts[i] : make_uint4(0u, 0u, 0u, 0u);
          }
#pragma unroll
          for (int u = 0; u < kTokBatch; ++u)
            if (i0 + u * 32 < a.L16) td[i0 + u * 32] = t4[u];
        }
      }
    }
    f = seg_end;
  }
}

// Grid size from the work: enough CTAs that each warp runs about `iters`
// iterations of its unrolled loop (`per_iter` units each), so the block
// scheduler balances the tail and a CTA that starts late (its SM still busy
// with another kernel) holds up little work; a small batch is spread over up
// to one wave (blocks resident per SM x SMs, queried once per kernel) with
// at least one iteration per warp.
template <typename Kern>
unsigned grid_for(Kern kern, uint64_t units, uint64_t per_iter, int iters, int sms) {
  static int per_sm = 0;  // per template instantiation
  if (!per_sm) {
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
    if (per_sm < 1) per_sm = 1;
  }
  const uint64_t wave = (uint64_t)per_sm * sms;
  const uint64_t warp_iters = (units + per_iter - 1) / per_iter;
  uint64_t blocks = (warp_iters + (uint64_t)kWarps * iters - 1) / ((uint64_t)kWarps * iters);
  if (blocks < wave) {
    const uint64_t most = (warp_iters + kWarps - 1) / kWarps;
    blocks = most < wave ? most : wave;
  }
  return (unsigned)(blocks ? blocks : 1);
}

}  // namespace

cudaError_t launch_deliver(edp_ctx *ctx, const int64_t *idx, uint32_t B,
                           const edp_batch *out, cudaStream_t s, const DrawUniform *draw) {
  Common c{};
  c.idx = idx;
  if (draw) {
    c.draw = 1;
    c.seed = draw->seed;
    c.round = draw->round;
    c.idx_out = draw->idx_out;
  }
  c.B = B;
  c.cap = ctx->cap;
  const uint64_t size = ctx->total < ctx->cap ? ctx->total : ctx->cap;
  c.oldest = (ctx->total - size) % ctx->cap;
  c.nvalid = size - ctx->defer;
  c.action = ctx->st.action;
  c.reward = ctx->st.reward;
  c.done = ctx->st.done;
  c.act_out = out->action;
  c.rew_out = out->reward;
  c.done_out = out->done;
  c.q = out->q;
  c.isw = out->isw;
  c.beta = out->beta;
  c.gsrc0 = out->gather_src[0];
  c.gdst0 = out->gather_dst[0];
  c.gsrc1 = out->gather_src[1];
  c.gdst1 = out->gather_dst[1];
  c.ctrl = ctx->ctrl;
  c.r1 = ctx->r1;
  c.r2 = ctx->r2;
  const int sms = ctx->coop_sms;
  const auto &cfg = ctx->cfg;
  if (cfg.transform == EDP_XFORM_STACK_F32) {
    StackArgs a{};
    a.frames = ctx->st.obs;
    a.F = (uint32_t)ctx->obs_bytes;
    a.W = a.F / 4;
    a.K = cfg.frame_stack;
    a.obs = (float *)out->obs;
    a.next = (float *)out->next_obs;
    a.U = a.K + (a.next ? 1 : 0);
    // equal pieces: the fewest that divide the frame's 16-byte runs and fit
    // a stage
    const uint32_t runs = a.F / 16;
    uint32_t np = (a.F + kPiece - 1) / kPiece;
    while (runs % np) ++np;
    const uint64_t staged_units = (uint64_t)B * a.U * np;
    const uint64_t staged_grid = (uint64_t)kStagedPerSm * sms;
    if (staged_units >= 2 * staged_grid) {
      return launch_pdl(k_deliver_stack_staged, dim3((unsigned)staged_grid),
                        dim3(kStagedThreads), s, c, a, np, a.F / np);
    }
    // a small batch: one span of one unrolled iteration per warp, one chunk
    // per CTA, and the collate CTA
    a.span = 32 * kStackUnroll;
    const uint64_t units = (uint64_t)B * a.U * a.W;
    const uint64_t chunks = (units + (uint64_t)kWarps * a.span - 1) / ((uint64_t)kWarps * a.span);
    if (chunks + 1 > 0x7FFFFFFFull) return cudaErrorInvalidValue;
    return launch_pdl(k_deliver_stack<kStackUnroll>, dim3((unsigned)(chunks + 1)),
                      dim3(kThreads), s, c, a);
  } else if (cfg.transform == EDP_XFORM_HWC_CHW_BF16) {
    ChwArgs a{};
    a.obs = ctx->st.obs;
    a.HW = cfg.obs_h * cfg.obs_w;
    a.out = (__nv_bfloat16 *)out->obs;
    const uint64_t units = (uint64_t)B * (a.HW / 8);
    constexpr uint64_t it = 32 * kHwcUnroll;
    switch (cfg.obs_c) {
      case 1: {
        auto kern = k_deliver_hwc<1, kHwcUnroll>;
        return launch_pdl(kern, dim3(grid_for(kern, units, it, kHwcIters, sms)),
                          dim3(kThreads), s, c, a);
      }
      case 2: {
        auto kern = k_deliver_hwc<2, kHwcUnroll>;
        return launch_pdl(kern, dim3(grid_for(kern, units, it, kHwcIters, sms)),
                          dim3(kThreads), s, c, a);
      }
      case 3: {
        auto kern = k_deliver_hwc<3, kHwcUnroll>;
        return launch_pdl(kern, dim3(grid_for(kern, units, it, kHwcIters, sms)),
                          dim3(kThreads), s, c, a);
      }
      default: {
        auto kern = k_deliver_hwc<4, kHwcUnroll>;
        return launch_pdl(kern, dim3(grid_for(kern, units, it, kHwcIters, sms)),
                          dim3(kThreads), s, c, a);
      }
    }
  } else {
    NormArgs a{};
    a.obs_h = ctx->st.obs;
    a.obs_c = ctx->cap_c ? ctx->st.host_obs : nullptr;
    a.tok_h = ctx->st.tokens;
    a.tok_c = ctx->cap_c ? ctx->st.host_tokens : nullptr;
    a.cap_h = ctx->cap_h;
    a.cap_c = ctx->cap_c ? ctx->cap_c : 1;
    a.total = ctx->total;
    a.size = size;
    a.F8 = (uint32_t)(ctx->obs_bytes / 8);
    a.HW8 = cfg.obs_h * cfg.obs_w / 8;
    a.L16 = (uint32_t)(ctx->tok_bytes / 16);
    for (int i = 0; i < 4; ++i) {
      a.mean[i] = ctx->nmean[i];
      a.s1[i] = ctx->ns1[i];
      a.s2[i] = ctx->ns2[i];
      a.sd[i] = ctx->nstd[i] > 0.f ? ctx->nstd[i] : 1.f;
      a.aa[i] = ctx->naff_a[i];
      a.ab[i] = ctx->naff_b[i];
    }
    a.fast = ctx->norm_fast;
    a.out = (__nv_bfloat16 *)out->obs;
    a.tok_out = out->tokens;
    const uint64_t units = (uint64_t)B * a.F8;
    auto kern = ctx->norm_affine ? k_deliver_norm<kNormUnroll, true>
                                 : k_deliver_norm<kNormUnroll, false>;
    return launch_pdl(kern, dim3(grid_for(kern, units, 32 * kNormUnroll, kNormIters, sms)),
                      dim3(kThreads), s, c, a);
  }
  return cudaGetLastError();
}

}  // namespace edp
