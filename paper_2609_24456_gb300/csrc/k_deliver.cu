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
// holds as many CTAs as that takes (several waves), so the block scheduler,
// or for the frame stack a work counter, balances the tail.  A warp walks
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
// loads in flight per lane (8 x 8 bytes) in the normalising delivery
constexpr int kNormUnroll = 8;

// unrolled rows per warp iteration and iterations per warp (chunk span) of
// each kernel; CTA slots per SM the frame-stack delivery leaves free
constexpr int kStackUnroll = 4, kStackIters = 3, kStackHeadroom = 2;
constexpr int kStackMinBlocks = 6;  // __launch_bounds__: at most 40 registers
constexpr int kHwcUnroll = 2, kHwcIters = 2;
constexpr int kNormIters = 3;

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
  unsigned long long *work;  // this launch's work word, or null (one chunk per CTA)
  unsigned long long work_tag;
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

// Importance weight (q_min / q_k)^beta in fp64, one rounding to fp32.
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
// Work claims of a persistent delivery grid.  The CTAs of a launch take
// chunks in order from one 64-bit work word of the context, laid out as
//   [63:28] owner tag   [27:0] chunks handed out;
// tag 0 means free.  A launch's tag is 1 + its call number on the context
// (host side: unique for every call, and for every node of a captured
// graph).  A CTA claims from the word if its launch owns it, takes the word
// over if it is free (claiming chunk 0), and otherwise -- another launch
// still owns it -- takes a fixed share: chunks blockIdx.x, blockIdx.x +
// gridDim.x, ...  A one-thread release kernel, queued after the delivery
// on the same stream, frees the word once every CTA of the launch has
// finished, so an owned word never changes hands while its owner runs, a
// replayed graph finds its words free again, and no claim of one launch
// can land on another's count.  Every chunk is processed: if any CTA of
// the launch owns the word, the owning CTAs claim until the chunks run out;
// if none does, the fixed shares cover them all; where both happen some
// chunks are written twice, with the same bytes.  (Only the same captured
// node running twice at once could meet its own tag on a live word; the
// two share the claims and, having the same arguments, still write every
// chunk of the one batch.)
// ---------------------------------------------------------------------------
constexpr int kWorkTagShift = 28;
constexpr unsigned long long kWorkClaimMask = (1ull << kWorkTagShift) - 1;
constexpr uint32_t kWorkMaxChunks = 1u << 27;  // chunks + grid stay below 2^28
constexpr uint32_t kWorkFixed = 0xffffffffu;   // first claim: take the fixed share
constexpr uint32_t kWorkDone = 0xfffffffeu;    // no chunk left for this launch

// A chunk of the launch with tag `tag` (or kWorkDone).
__device__ __forceinline__ uint32_t work_claim(unsigned long long *wd,
                                               unsigned long long tag) {
  const unsigned long long old = atomicAdd(wd, 1ull);
  return (old >> kWorkTagShift) == tag ? (uint32_t)(old & kWorkClaimMask) : kWorkDone;
}

// A CTA's first claim: a chunk, or kWorkFixed when another launch owns the
// word.
__device__ __forceinline__ uint32_t work_first(unsigned long long *wd,
                                               unsigned long long tag) {
  unsigned long long w = *reinterpret_cast<volatile unsigned long long *>(wd);
  for (int tries = 0; tries < 8; ++tries) {
    const unsigned long long owner = w >> kWorkTagShift;
    if (owner == tag) return work_claim(wd, tag);
    if (owner != 0) return kWorkFixed;
    const unsigned long long mine = (tag << kWorkTagShift) | 1ull;  // chunk 0 taken
    const unsigned long long prev = atomicCAS(wd, w, mine);
    if (prev == w) return 0;
    w = prev;
  }
  return kWorkFixed;
}

// Frees the word of the launch with tag `tag`, after that launch (the
// preceding kernel on the stream) has completed.
__global__ void k_work_release(unsigned long long *wd, unsigned long long tag) {
  pdl_wait();
  pdl_launch();
  unsigned long long w = *reinterpret_cast<volatile unsigned long long *>(wd);
  for (int tries = 0; tries < 8 && (w >> kWorkTagShift) == tag; ++tries) {
    const unsigned long long prev = atomicCAS(wd, w, 0ull);
    if (prev == w) break;
    w = prev;
  }
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
// Scheduling: the work is cut into chunks of kWarps spans.  A batch with
// more chunks than the grid holds runs on a persistent grid that leaves
// kStackHeadroom CTA slots of every SM free -- so the small sampling and
// priority-update kernels of the next round find room beside a running
// delivery (the overlapped timing of Sec. 6.1) -- and its CTAs claim chunks
// from a work word (above) until the batch is done, which balances the
// tail without relying on all CTAs being resident.  A smaller batch
// runs one chunk per CTA with no counter, and one more CTA collates the
// whole batch (collate_batch) so that no streaming warp waits on it; on the
// persistent grid the head warp of each sample collates it before its span
// (measured: a collate CTA there made the isolated launch faster, 29.1 ->
// 25.6 us, but the overlapped replay round slower, 21.0 -> 23-24 us).
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
                                           uint64_t pol, bool head_collate) {
  const uint64_t per = (uint64_t)a.U * a.W;  // units per sample
  const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
  while (f < end) {
    const uint32_t k = (uint32_t)(f / per);
    const uint32_t rem = (uint32_t)(f - (uint64_t)k * per);
    const uint32_t m = rem / a.W;
    const uint32_t w_lo = rem - m * a.W;
    const uint64_t seg_end = min(end, (uint64_t)k * per + (uint64_t)(m + 1) * a.W);
    const uint32_t w_hi = (uint32_t)(seg_end - (uint64_t)k * per - (uint64_t)m * a.W);
    const bool head = head_collate && rem == 0;
    uint64_t slot = 0, off = 0;
    const bool ok = sample_slot(c, k, &slot, &off, head && lane == 0);
    if (head) collate(c, k, ok, slot, off, lane);
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
  __shared__ uint32_t s_chunk[2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint64_t pol = policy_stream();
  pdl_wait();
  pdl_launch();
  const uint64_t total = (uint64_t)c.B * a.U * a.W;
  const uint64_t per_chunk = (uint64_t)kWarps * a.span;
  if (!c.work) {  // one chunk per CTA; CTA 0 collates the batch
    if (blockIdx.x == 0) {
      collate_batch(c);
      return;
    }
    const uint64_t f = (uint64_t)(blockIdx.x - 1) * per_chunk + (uint64_t)warp * a.span;
    if (f < total) stack_span<UN>(c, a, f, min(total, f + a.span), lane, pol, false);
    return;
  }
  // Thread 0 makes the CTA's first claim (or takes the fixed share), grabs
  // the next chunk while the CTA works on the current one and publishes it
  // in the other half of s_chunk before the one barrier per chunk; the half
  // it overwrites was read before the previous barrier.
  __shared__ uint32_t s_owned;
  if (threadIdx.x == 0) {
    const uint32_t first = work_first(c.work, c.work_tag);
    s_owned = first != kWorkFixed;
    s_chunk[0] = first != kWorkFixed ? first : blockIdx.x;
  }
  __syncthreads();
  const bool owned = s_owned != 0;
  uint32_t cur = s_chunk[0];
  for (int p = 1;; p ^= 1) {
    const uint64_t f0 = (uint64_t)cur * per_chunk;
    if (f0 >= total) break;  // uniform across the CTA
    uint32_t nxt = 0;
    if (threadIdx.x == 0) nxt = owned ? work_claim(c.work, c.work_tag) : cur + gridDim.x;
    const uint64_t f = f0 + (uint64_t)warp * a.span;
    if (f < total) stack_span<UN>(c, a, f, min(total, f + a.span), lane, pol, true);
    if (threadIdx.x == 0) s_chunk[p] = nxt;
    __syncthreads();
    cur = s_chunk[p];
  }
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
      if (a.tok_out) {
        const uint4 *ts = reinterpret_cast<const uint4 *>(
            (hbm ? a.tok_h : a.tok_c) + ps * a.L16 * 4ull);
        uint4 *td = reinterpret_cast<uint4 *>(a.tok_out + (uint64_t)k * a.L16 * 4ull);
        for (uint32_t i = lane; i < a.L16; i += 32)
          td[i] = ok ? ts[i] : make_uint4(0u, 0u, 0u, 0u);
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
    const uint64_t units = (uint64_t)B * a.U * a.W;
    auto kern = k_deliver_stack<kStackUnroll>;
    static int per_sm = 0;
    if (!per_sm) {
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
      if (per_sm < 1) per_sm = 1;
    }
    const int resident = per_sm > kStackHeadroom ? per_sm - kStackHeadroom : 1;
    uint64_t grid = (uint64_t)resident * sms;
    auto n_chunks = [&](uint32_t span) {
      return (units + (uint64_t)kWarps * span - 1) / ((uint64_t)kWarps * span);
    };
    a.span = 32 * kStackUnroll * kStackIters;
    uint64_t chunks = n_chunks(a.span);
    if (chunks < grid) {  // a small batch: one iteration per warp, more CTAs
      a.span = 32 * kStackUnroll;
      chunks = n_chunks(a.span);
    }
    if (grid >= chunks || chunks + grid >= kWorkMaxChunks) {
      grid = chunks + 1;  // one chunk per CTA and the collate CTA, no work word
      if (grid > 0x7FFFFFFFull) return cudaErrorInvalidValue;
      return launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), s, c, a);
    }
    const uint64_t seq = ctx->work_seq++;
    c.work = ctx->ctrl->work + (seq % kWorkSlots);
    c.work_tag = seq % ((1ull << (64 - kWorkTagShift)) - 1) + 1;
    cudaError_t e = launch_pdl(kern, dim3((unsigned)grid), dim3(kThreads), s, c, a);
    if (e != cudaSuccess) return e;
    return launch_pdl(k_work_release, dim3(1), dim3(32), s, c.work, c.work_tag);
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
