// k_deliver.cu -- fused delivery: gather the sampled transitions, transform
// their uint8 payload into the learner layout, collate metadata, and
// compute importance weights, in one pass over the payload (Sec. 2.2:
// delivery "materializes the selected transitions and performs batch/layout
// transformations").
//
// Work decomposition: the batch's output is a flat sequence of units (a
// 32-bit word of a frame, an 8-pixel group, an 8-byte run of a plane).  The
// grid is one wave of persistent CTAs (occupancy x SMs) and each warp takes
// one contiguous, equal span of that sequence, so every SM finishes at the
// same time.  A warp walks its span segment by segment (a segment never
// crosses a frame or image), resolving the sample's slot, episode-boundary
// mask and source pointer once per segment.  Loads are the payload bytes a
// lane needs for one 16-byte output store, so every warp-wide store
// instruction writes 512 contiguous bytes.  The byte->float step is
// x = b (exact), fl32(b/255) = fma(x, r1, x*r2) with one rounding (see
// unit_f32), then optionally the per-channel normalisation and the
// round-to-nearest-even bfloat16 conversion.
//
// This kernel is HBM-bound: per sample it reads the unique source bytes once
// and writes the (2-4x larger) float output once.
#include "edp_internal.cuh"

namespace edp {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
// loads in flight per lane (8 x 8 bytes) in the normalising delivery
constexpr int kNormUnroll = 8;

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
};

// Resolve slot -> logical offset; false (and a flag) when not sampleable.
__device__ __forceinline__ bool sample_slot(const Common &c, uint32_t k,
                                            uint64_t *slot, uint64_t *off,
                                            bool report) {
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
    if (lane == 0) {
      const uint32_t qk = c.q[k];
      float w = 0.f;
      if (qk == m) {
        w = 1.f;
      } else if (qk) {
        // m / qk with an fp32 seed and two Newton steps (no fp64 divide)
        const double d = (double)qk;
        double y = (double)(1.0f / (float)qk);
        y = fma(y, fma(-d, y, 1.0), y);
        y = fma(y, fma(-d, y, 1.0), y);
        w = (float)pow_pos<false>((double)m * y, c.beta);
      }
      c.isw[k] = w;
    }
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
// Frame stack, float32 (DQN), on the bulk-copy engine.  A unit is one part
// (<= 2400 bytes) of frame m in [0, K] of sample k -- the frame at logical
// offset j = off - K + 1 + m, which is obs slot m (m < K) and next_obs slot
// m - 1 (m >= 1).  Each persistent CTA owns a contiguous range of units and
// runs a kStages-deep pipeline over it:
//   thread 0  bulk-loads the part of unit i + kStages - 1 into its stage
//             (mbarrier with transaction count; units needing no load arrive
//             on the barrier without bytes so the phases stay in step);
//   all       wait for unit i's stage, convert its bytes to fp32 in shared
//             memory, fence the async proxy;
//   thread 0  bulk-stores the fp32 tile to obs and/or next_obs (a zero tile
//             for zero-padded frames) and commits one store group per unit;
//             before a stage's tile is rewritten, at most kStages - 1 groups
//             may still be reading shared memory.
// The per-unit control (slot, episode-boundary mask, source and destination
// offsets) is resolved for 256 units at a time, one thread per unit, before
// the pipeline; the head unit of each sample also runs the collate.
// ---------------------------------------------------------------------------
constexpr int kStages = 4;
constexpr int kCtlUnits = 256;

struct StackArgs {
  const uint8_t *frames;
  uint32_t F;     // bytes per frame
  uint32_t K;
  uint32_t U;     // frames per sample (K, or K + 1 with next_obs)
  uint32_t P;     // parts per frame
  uint32_t part;  // bytes per part (multiple of 16; the last may be shorter)
  float *obs;
  float *next;
};

struct UnitCtl {
  uint64_t src;    // byte offset of the part in the frame ring
  uint64_t dobs;   // float offset in obs, or ~0
  uint64_t dnext;  // float offset in next_obs, or ~0
  uint32_t bytes;  // bytes of this part
  uint32_t flags;  // kLoad | kZeroObs | kZeroNext
};
constexpr uint32_t kLoad = 1u, kZeroObs = 2u, kZeroNext = 4u;

__host__ __device__ constexpr size_t align_up(size_t x, size_t a) {
  return (x + a - 1) / a * a;
}
// shared memory: barriers | control | kStages input parts | kStages fp32
// tiles | one zero tile
__host__ __device__ inline size_t stack_smem(uint32_t part) {
  return 128 + align_up(kCtlUnits * sizeof(UnitCtl), 128) +
         align_up((size_t)kStages * part, 128) + (size_t)kStages * part * 4 +
         (size_t)part * 4;
}

__global__ void __launch_bounds__(kThreads)
k_deliver_stack(Common c, StackArgs a) {
  extern __shared__ __align__(128) uint8_t sm[];
  uint64_t *bar = reinterpret_cast<uint64_t *>(sm);
  UnitCtl *ctl = reinterpret_cast<UnitCtl *>(sm + 128);
  uint8_t *in = sm + 128 + align_up(kCtlUnits * sizeof(UnitCtl), 128);
  float *tile = reinterpret_cast<float *>(in + align_up((size_t)kStages * a.part, 128));
  float *zero = tile + (size_t)kStages * a.part;
  __shared__ int s_abort;  // a bounded wait expired: stop the pipeline
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const uint64_t pol = policy_stream();
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
    s_abort = 0;
  }
  for (uint32_t i = tid; i < a.part; i += kThreads) zero[i] = 0.f;
  pdl_wait();
  pdl_launch();
  fence_proxy_async();
  __syncthreads();

  const uint64_t total = (uint64_t)c.B * a.U * a.P;
  const uint64_t per = (total + gridDim.x - 1) / gridDim.x;
  const uint64_t u0 = (uint64_t)blockIdx.x * per;
  const uint64_t u1 = min(total, u0 + per);
  uint32_t it = 0;  // pipeline position across control batches
  for (uint64_t ub = u0; ub < u1; ub += kCtlUnits) {
    const uint32_t nu = (uint32_t)min((uint64_t)kCtlUnits, u1 - ub);
    // ---- control, one thread per unit
    for (uint32_t t = tid; t < nu; t += kThreads) {
      const uint64_t u = ub + t;
      const uint32_t k = (uint32_t)(u / (a.U * a.P));
      const uint32_t rem = (uint32_t)(u % (a.U * a.P));
      const uint32_t m = rem / a.P, p = rem % a.P;
      uint64_t slot = 0, off = 0;
      const bool ok = sample_slot(c, k, &slot, &off, m == 0 && p == 0);
      const int64_t j = (int64_t)off - (int64_t)(a.K - 1) + (int64_t)m;
      // an episode end at offsets [j, off - 1] zeroes the frame in obs,
      // one at [j, off] in next_obs
      bool end_before = false, end_at = false;
      if (ok && j >= 0) {
        for (int64_t o = j; o <= (int64_t)off; ++o) {
          const uint64_t t2 = c.oldest + (uint64_t)o;
          const bool d = c.done[t2 >= c.cap ? t2 - c.cap : t2] != 0;
          if (o < (int64_t)off) end_before |= d; else end_at = d;
        }
      }
      const bool has_obs = m < a.K;
      const bool has_next = a.next && m >= 1;
      const bool zo = !ok || j < 0 || end_before;
      const bool zn = !ok || j < 0 || end_before || end_at;
      UnitCtl e;
      e.bytes = p + 1 < a.P ? a.part : a.F - (a.P - 1) * a.part;
      const uint64_t js = c.oldest + (uint64_t)(j < 0 ? 0 : j);
      e.src = (js >= c.cap ? js - c.cap : js) * a.F + (uint64_t)p * a.part;
      e.dobs = has_obs ? ((uint64_t)k * a.K + m) * a.F + (uint64_t)p * a.part : ~0ull;
      e.dnext = has_next ? ((uint64_t)k * a.K + m - 1) * a.F + (uint64_t)p * a.part : ~0ull;
      e.flags = ((has_obs && !zo) || (has_next && !zn) ? kLoad : 0u) |
                (zo ? kZeroObs : 0u) | (zn ? kZeroNext : 0u);
      ctl[t] = e;
    }
    __syncthreads();
    // ---- bulk loads of the first kStages - 1 units
    if (tid == 0)
      for (uint32_t i = 0; i + 1 < kStages && i < nu; ++i) {
        const UnitCtl &e = ctl[i];
        const uint32_t st = (it + i) % kStages;
        if (e.flags & kLoad) {
          mbar_expect_tx(&bar[st], e.bytes);
          tma_load(in + (size_t)st * a.part, a.frames + e.src, e.bytes, &bar[st], pol);
        } else {
          mbar_expect_tx(&bar[st], 0);
        }
      }
    // ---- collate of the samples whose head unit is in this batch
    for (uint32_t t = warp; t < nu; t += kWarps) {
      const uint64_t u = ub + t;
      if (u % ((uint64_t)a.U * a.P) != 0) continue;
      const uint32_t k = (uint32_t)(u / (a.U * a.P));
      uint64_t slot = 0, off = 0;
      const bool ok = sample_slot(c, k, &slot, &off, false);
      collate(c, k, ok, slot, off, lane);
    }
    // ---- pipeline
    for (uint32_t i = 0; i < nu; ++i, ++it) {
      const uint32_t st = it % kStages;
      if (tid == 0 && i + kStages - 1 < nu) {
        const UnitCtl &e = ctl[i + kStages - 1];
        const uint32_t sn = (it + kStages - 1) % kStages;
        if (e.flags & kLoad) {
          mbar_expect_tx(&bar[sn], e.bytes);
          tma_load(in + (size_t)sn * a.part, a.frames + e.src, e.bytes, &bar[sn], pol);
        } else {
          mbar_expect_tx(&bar[sn], 0);
        }
      }
      const UnitCtl e = ctl[i];
      if (!mbar_wait(&bar[st], (it / kStages) & 1u, c.ctrl)) s_abort = 1;
      if (tid == 0) tma_wait_read<kStages - 1>();  // tile st is free again
      __syncthreads();
      if (s_abort) break;
      float4 *tl = reinterpret_cast<float4 *>(tile + (size_t)st * a.part);
      if (e.flags & kLoad) {
        const uint32_t *src = reinterpret_cast<const uint32_t *>(in + (size_t)st * a.part);
        for (uint32_t w = tid; w < e.bytes / 4; w += kThreads) {
          const uint32_t v = src[w];
          float4 fv;
          fv.x = unit_f32(byte_f(v, 0), c.r1, c.r2);
          fv.y = unit_f32(byte_f(v, 1), c.r1, c.r2);
          fv.z = unit_f32(byte_f(v, 2), c.r1, c.r2);
          fv.w = unit_f32(byte_f(v, 3), c.r1, c.r2);
          tl[w] = fv;
        }
      }
      fence_proxy_async();
      __syncthreads();
      if (tid == 0) {
        if (e.dobs != ~0ull)
          tma_store(a.obs + e.dobs, (e.flags & kZeroObs) ? zero : (float *)tl,
                    e.bytes * 4, pol);
        if (e.dnext != ~0ull)
          tma_store(a.next + e.dnext, (e.flags & kZeroNext) ? zero : (float *)tl,
                    e.bytes * 4, pol);
        tma_commit();
      }
    }
    __syncthreads();  // the control table is rewritten by the next batch
    if (s_abort) break;
  }
  if (tid == 0) tma_wait_all();
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
  int fast;
  __nv_bfloat16 *out;
  int32_t *tok_out;
};

template <int UN>
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
        const float mc = a.mean[ch], s1 = a.s1[ch], s2 = a.s2[ch];
        float fv[8];
#pragma unroll
        for (int bb = 0; bb < 8; ++bb) {
          const float x = unit_f32(byte_f(bb < 4 ? v[u].x : v[u].y, bb & 3), c.r1, c.r2);
          const float tt = __fsub_rn(x, mc);
          fv[bb] = a.fast ? __fmaf_rn(tt, s1, __fmul_rn(tt, s2)) : __fdiv_rn(tt, a.sd[ch]);
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

// One wave of persistent CTAs: blocks resident per SM x SMs (queried once
// per kernel), never more CTAs than there are 32-unit rows of work.
template <typename Kern>
unsigned one_wave(Kern kern, uint64_t total_units, int sms) {
  static int per_sm = 0;  // per template instantiation
  if (!per_sm) {
    cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, kThreads, 0);
    if (per_sm < 1) per_sm = 1;
  }
  const uint64_t rows = (total_units + 31) / 32;
  uint64_t blocks = (uint64_t)per_sm * sms;
  const uint64_t need = (rows + kWarps - 1) / kWarps;
  if (blocks > need) blocks = need;
  return (unsigned)(blocks ? blocks : 1);
}

}  // namespace

cudaError_t launch_deliver(edp_ctx *ctx, const int64_t *idx, uint32_t B,
                           const edp_batch *out, cudaStream_t s) {
  Common c{};
  c.idx = idx;
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
    a.K = cfg.frame_stack;
    a.obs = (float *)out->obs;
    a.next = (float *)out->next_obs;
    a.U = a.K + (a.next ? 1 : 0);
    // parts of at most ~2.4 KB, each a multiple of 16 bytes
    a.P = (a.F + 2399) / 2400;
    a.part = (uint32_t)(((a.F / 16) + a.P - 1) / a.P * 16);
    a.P = (a.F + a.part - 1) / a.part;
    const size_t smem = stack_smem(a.part);
    static int per_sm = 0;
    static size_t smem_set = 0;
    if (smem_set != smem) {
      cudaFuncSetAttribute(k_deliver_stack, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           (int)smem);
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k_deliver_stack, kThreads, smem);
      if (per_sm < 1) per_sm = 1;
      smem_set = smem;
    }
    const uint64_t units = (uint64_t)B * a.U * a.P;
    uint64_t grid = (uint64_t)per_sm * sms;
    if (grid > units) grid = units;
    cudaLaunchConfig_t lc = {};
    lc.gridDim = dim3((unsigned)grid);
    lc.blockDim = dim3(kThreads);
    lc.dynamicSmemBytes = smem;
    lc.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    lc.attrs = attr;
    lc.numAttrs = 1;
    return cudaLaunchKernelEx(&lc, k_deliver_stack, c, a);
  } else if (cfg.transform == EDP_XFORM_HWC_CHW_BF16) {
    ChwArgs a{};
    a.obs = ctx->st.obs;
    a.HW = cfg.obs_h * cfg.obs_w;
    a.out = (__nv_bfloat16 *)out->obs;
    const uint64_t units = (uint64_t)B * (a.HW / 8);
    switch (cfg.obs_c) {
      case 1:
        return launch_pdl(k_deliver_hwc<1, 2>, dim3(one_wave(k_deliver_hwc<1, 2>, units, sms)),
                          dim3(kThreads), s, c, a);
      case 2:
        return launch_pdl(k_deliver_hwc<2, 2>, dim3(one_wave(k_deliver_hwc<2, 2>, units, sms)),
                          dim3(kThreads), s, c, a);
      case 3:
        return launch_pdl(k_deliver_hwc<3, 2>, dim3(one_wave(k_deliver_hwc<3, 2>, units, sms)),
                          dim3(kThreads), s, c, a);
      default:
        return launch_pdl(k_deliver_hwc<4, 2>, dim3(one_wave(k_deliver_hwc<4, 2>, units, sms)),
                          dim3(kThreads), s, c, a);
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
    }
    a.fast = ctx->norm_fast;
    a.out = (__nv_bfloat16 *)out->obs;
    a.tok_out = out->tokens;
    const uint64_t units = (uint64_t)B * a.F8;
    return launch_pdl(k_deliver_norm<kNormUnroll>,
                      dim3(one_wave(k_deliver_norm<kNormUnroll>, units, sms)),
                      dim3(kThreads), s, c, a);
  }
  return cudaGetLastError();
}

}  // namespace edp
