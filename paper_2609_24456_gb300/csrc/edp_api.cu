// edp_api.cu -- the C ABI of libedp: argument validation, host-side cursors
// of the logical ring, and kernel dispatch.  Every step of the data path
// runs in the kernels of the other translation units.
#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <initializer_list>
#include <new>

#include "edp_internal.cuh"

using namespace edp;

namespace {

void *default_alloc(void *, size_t bytes) {
  void *p = nullptr;
  if (cudaMalloc(&p, bytes) != cudaSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return p;
}

void default_free(void *, void *p) { cudaFree(p); }

edp_status cuda_fail(edp_ctx *c, cudaError_t e, const char *where) {
  return fail(c, EDP_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

edp_status create_fail(edp_ctx *c, const char *fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  fprintf(stderr, "edp_create: %s\n", buf);
  delete c;
  return EDP_ERR_INVALID;
}

bool aligned16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

uint64_t ring_size(const edp_ctx *c) { return c->total < c->cap ? c->total : c->cap; }

uint64_t n_valid(const edp_ctx *c) {
  const uint64_t s = ring_size(c);
  return s >= (uint64_t)c->defer ? s - c->defer : 0;
}

void free_all(edp_ctx *c) {
  edp_free_fn fr = c->cfg.free ? c->cfg.free : default_free;
  if (c->tree_mem) fr(c->cfg.alloc_user, c->tree_mem);
  if (c->ctrl) fr(c->cfg.alloc_user, c->ctrl);
  if (c->scratch) fr(c->cfg.alloc_user, c->scratch);
  if (c->qbuf) fr(c->cfg.alloc_user, c->qbuf);
  if (c->perm_scratch) fr(c->cfg.alloc_user, c->perm_scratch);
  c->qbuf = nullptr;
  c->perm_scratch = nullptr;
  c->tree_mem = nullptr;
  c->ctrl = nullptr;
  c->scratch = nullptr;
}

// Host self-check of the transform constants against IEEE division (the
// device evaluates exactly these operations).
bool unit_constants(float *r1, float *r2) {
  *r1 = 1.0f / 255.0f;
  *r2 = (float)(1.0 / 255.0 - (double)*r1);
  for (int b = 0; b < 256; ++b) {
    const float x = (float)b;
    const float ref = x / 255.0f;
    const float got = fmaf(x, *r1, x * *r2);
    if (got != ref) return false;
  }
  return true;
}

bool norm_constants(edp_ctx *c) {
  bool fast = true;
  for (uint32_t ch = 0; ch < c->cfg.obs_c; ++ch) {
    const float m = c->cfg.norm_mean[ch], s = c->cfg.norm_std[ch];
    const float s1 = (float)(1.0 / (double)s);
    const float s2 = (float)(1.0 / (double)s - (double)s1);
    c->nmean[ch] = m;
    c->nstd[ch] = s;
    c->ns1[ch] = s1;
    c->ns2[ch] = s2;
    for (int b = 0; b < 256; ++b) {
      const float x = (float)b / 255.0f;
      const float t = x - m;
      if (fmaf(t, s1, t * s2) != t / s) fast = false;
    }
  }
  return fast;
}

// bfloat16 bits of a finite float, rounded to nearest even (the device's
// conversion).
uint16_t bf16_rne(float f) {
  uint32_t u;
  std::memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

float ulp_step(float x, int d) {
  for (; d > 0; --d) x = std::nextafter(x, INFINITY);
  for (; d < 0; ++d) x = std::nextafter(x, -INFINITY);
  return x;
}

// The normalised bf16 of byte b in channel c is a function of (b, c) alone:
// bf16(fl32(fl32(fl32(b/255) - mean_c) / std_c)).  One FMA,
// bf16(fma(b, A_c, B_c)), reproduces it for all 256 bytes when A_c and B_c
// are close enough to 1/(255 std_c) and -mean_c/std_c and no result of the
// chain sits on a bf16 rounding boundary the FMA crosses; the constants are
// searched within kAffineUlps ulps of those values (nearest first) and every
// byte is checked.  False when some channel has no such pair.
constexpr int kAffineUlps = 16;

bool norm_affine_constants(edp_ctx *c) {
  for (uint32_t ch = 0; ch < c->cfg.obs_c; ++ch) {
    const float m = c->cfg.norm_mean[ch], s = c->cfg.norm_std[ch];
    uint16_t want[256];
    for (int b = 0; b < 256; ++b) {
      const float x = (float)b / 255.0f;
      const float t = x - m;
      want[b] = bf16_rne(t / s);
    }
    const float a0 = (float)(1.0 / (255.0 * (double)s));
    const float b0 = (float)(-(double)m / (double)s);
    if (!std::isfinite(a0) || !std::isfinite(b0)) return false;
    bool found = false;
    for (int r = 0; r <= kAffineUlps && !found; ++r)
      for (int da = -r; da <= r && !found; ++da)
        for (int db = -r; db <= r && !found; ++db) {
          if (std::max(std::abs(da), std::abs(db)) != r) continue;
          const float A = ulp_step(a0, da), B = ulp_step(b0, db);
          bool ok = std::isfinite(A) && std::isfinite(B);
          for (int b = 0; b < 256 && ok; ++b) ok = bf16_rne(std::fma((float)b, A, B)) == want[b];
          if (ok) {
            c->naff_a[ch] = A;
            c->naff_b[ch] = B;
            found = true;
          }
        }
    if (!found) return false;
  }
  return true;
}

}  // namespace

edp_status edp::fail(edp_ctx *c, edp_status s, const char *fmt, ...) {
  if (c) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    c->err = buf;
  }
  return s;
}

bool edp::device_view(const edp_ctx *c, const void *p, const void **out,
                      bool allow_host) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (a.type == cudaMemoryTypeDevice || a.type == cudaMemoryTypeManaged) {
    if (a.device != c->cfg.device) return false;
    *out = p;
    return true;
  }
  if (a.type == cudaMemoryTypeHost && allow_host && a.devicePointer) {
    *out = a.devicePointer;
    return true;
  }
  return false;
}

bool edp::host_memory(const void *p) {
  if (!p) return false;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  return a.type == cudaMemoryTypeHost;
}

namespace {
// Traffic counters: bytes at p (device or page-locked host memory).
void count_read(edp_ctx *c, const void *p, uint64_t bytes) {
  if (p && bytes) (host_memory(p) ? c->cnt.link_read : c->cnt.hbm_read) += bytes;
}
void count_write(edp_ctx *c, const void *p, uint64_t bytes) {
  if (p && bytes) (host_memory(p) ? c->cnt.link_write : c->cnt.hbm_write) += bytes;
}
// Device-resident arrays of a call (index, priority and scalar arrays).
void count_hbm(edp_ctx *c, uint64_t read, uint64_t write) {
  c->cnt.hbm_read += read;
  c->cnt.hbm_write += write;
  ++c->cnt.calls;
}
}  // namespace

edp_status edp::launch_fail(edp_ctx *c, cudaError_t e, const char *where) {
  if (e == cudaErrorMemoryAllocation)
    return fail(c, EDP_ERR_OOM, "%s: scratch allocation failed", where);
  if (e == cudaErrorStreamCaptureUnsupported)
    return fail(c, EDP_ERR_STATE,
                "%s: not allowed while the stream is being captured (its scratch "
                "would have to grow: make one call of this size before capture)",
                where);
  return fail(c, EDP_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
}

edp_status edp::update_args(edp_ctx *ctx, const char *who, const int64_t *idx,
                            const uint32_t *q, const float *td, uint32_t n,
                            double alpha, double eps) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!ctx->depth) return fail(ctx, EDP_ERR_STATE, "%s: context has no priorities", who);
  if (n == 0) return EDP_OK;
  if (!idx || (!q && !td)) return fail(ctx, EDP_ERR_INVALID, "%s: NULL input", who);
  const void *p;
  if (!device_view(ctx, idx, &p, false) || (q && !device_view(ctx, q, &p, false)) ||
      (td && !device_view(ctx, td, &p, false)))
    return fail(ctx, EDP_ERR_INVALID, "%s: inputs must be device memory", who);
  if (td && !(alpha >= 0.0 && eps >= 0.0))
    return fail(ctx, EDP_ERR_INVALID, "%s: alpha, eps >= 0", who);
  return EDP_OK;
}

namespace {

// Grow-only block (*blk, *have bytes) to at least `want` bytes; the first
// `zero_head` bytes of a new block are zeroed.
cudaError_t grow(edp_ctx *ctx, void **blk, size_t *have, size_t want, size_t zero_head,
                 cudaStream_t s) {
  if (want <= *have) return cudaSuccess;
  cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
  if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) {
    cudaGetLastError();  // e.g. the legacy stream while another captures
    return cudaErrorStreamCaptureUnsupported;
  }
  if (cs != cudaStreamCaptureStatusNone) return cudaErrorStreamCaptureUnsupported;
  edp_alloc_fn al = ctx->cfg.alloc ? ctx->cfg.alloc : default_alloc;
  edp_free_fn fr = ctx->cfg.free ? ctx->cfg.free : default_free;
  if (*blk) {
    cudaDeviceSynchronize();  // the old block may still be in use
    fr(ctx->cfg.alloc_user, *blk);
    *blk = nullptr;
    *have = 0;
  }
  want = (want + 255) & ~(size_t)255;
  void *p = al(ctx->cfg.alloc_user, want);
  if (!p) return cudaErrorMemoryAllocation;
  if (zero_head && cudaMemset(p, 0, zero_head) != cudaSuccess) {
    cudaGetLastError();
    fr(ctx->cfg.alloc_user, p);
    return cudaErrorMemoryAllocation;
  }
  *blk = p;
  *have = want;
  return cudaSuccess;
}

}  // namespace

cudaError_t edp::ctx_scratch(edp_ctx *ctx, size_t bytes, cudaStream_t s, void **out) {
  const cudaError_t e = grow(ctx, &ctx->scratch, &ctx->scratch_bytes, bytes, 0, s);
  *out = ctx->scratch;
  return e;
}

cudaError_t edp::ctx_perm_scratch(edp_ctx *ctx, size_t bytes, cudaStream_t s, void **out) {
  const cudaError_t e =
      grow(ctx, &ctx->perm_scratch, &ctx->perm_bytes, bytes, perm_zeroed_bytes(), s);
  *out = ctx->perm_scratch;
  return e;
}

cudaError_t edp::ctx_qbuf(edp_ctx *ctx, size_t n, cudaStream_t s, uint32_t **out) {
  void *blk = ctx->qbuf;
  size_t have = ctx->qbuf_n * 4;
  const cudaError_t e = grow(ctx, &blk, &have, (n < 4096 ? 4096 : n) * 4, 0, s);
  ctx->qbuf = (uint32_t *)blk;
  ctx->qbuf_n = have / 4;
  *out = ctx->qbuf;
  return e;
}

extern "C" {

int edp_abi_version(void) { return EDP_ABI_VERSION; }

const char *edp_last_error(const edp_ctx *ctx) {
  return ctx ? ctx->err.c_str() : "null context";
}

edp_status edp_create(const edp_config *cfg, const edp_storage *st,
                      edp_ctx **out) {
  if (!cfg || !st || !out) return EDP_ERR_INVALID;
  *out = nullptr;
  edp_ctx *c = new (std::nothrow) edp_ctx();
  if (!c) return EDP_ERR_OOM;
  c->cfg = *cfg;
  c->st = *st;
#define bad(...) create_fail(c, __VA_ARGS__)
  for (int i = 0; i < 7; ++i)
    if (cfg->reserved[i]) return bad("reserved fields must be 0");
  if (cfg->capacity == 0 || cfg->capacity > 0xFFFFFFFFull)
    return bad("capacity must be in [1, 2^32-1]");
  if (cfg->hbm_capacity == 0 || cfg->hbm_capacity > cfg->capacity)
    return bad("hbm_capacity must be in [1, capacity]");
  if (!cfg->obs_c || !cfg->obs_h || !cfg->obs_w) return bad("empty obs shape");
  const uint64_t ob = (uint64_t)cfg->obs_c * cfg->obs_h * cfg->obs_w;
  if (ob % 16) return bad("obs bytes (%llu) must be a multiple of 16",
                          (unsigned long long)ob);
  if (ob > 0x7FFFFFFFull) return bad("obs too large");
  if (cfg->tokens % 4) return bad("tokens must be a multiple of 4");
  if (cfg->transform > EDP_XFORM_CHW_NORM_BF16) return bad("bad transform");
  const uint64_t hw = (uint64_t)cfg->obs_h * cfg->obs_w;
  if (cfg->transform == EDP_XFORM_STACK_F32) {
    if (cfg->obs_c != 1) return bad("STACK_F32 stores single-channel frames");
    if (cfg->frame_stack < 1 || cfg->frame_stack > 16)
      return bad("frame_stack must be in [1, 16]");
    if (!st->done) return bad("STACK_F32 needs the done field");
  } else {
    if (cfg->frame_stack != 1) return bad("frame_stack must be 1");
    if (cfg->next_obs) return bad("next_obs only with STACK_F32");
    if (cfg->obs_c > 4) return bad("obs_c must be <= 4");
    if (hw % 16) return bad("obs_h*obs_w must be a multiple of 16");
  }
  if (cfg->transform == EDP_XFORM_CHW_NORM_BF16)
    for (uint32_t ch = 0; ch < cfg->obs_c; ++ch)
      if (!(cfg->norm_std[ch] > 0.f) || !std::isfinite(cfg->norm_mean[ch]))
        return bad("norm_std must be > 0 and norm_mean finite");
  const bool tiered = cfg->hbm_capacity < cfg->capacity;
  if (tiered && cfg->transform != EDP_XFORM_CHW_NORM_BF16)
    return bad("the two-tier ring serves CHW_NORM_BF16 payloads");

  int ndev = 0;
  if (cudaGetDeviceCount(&ndev) != cudaSuccess || cfg->device < 0 ||
      cfg->device >= ndev) {
    cudaGetLastError();
    return bad("no CUDA device %d", cfg->device);
  }
  DeviceGuard dg(cfg->device);
  EDP_TRACE(__func__);
  if (!dg.ok()) return bad("cudaSetDevice failed");
  c->cap = cfg->capacity;
  c->cap_h = cfg->hbm_capacity;
  c->cap_c = cfg->capacity - cfg->hbm_capacity;
  c->obs_bytes = ob;
  c->tok_bytes = (uint64_t)cfg->tokens * 4;
  c->defer = cfg->next_obs ? 1 : 0;

  // storage pointers
  const void *p;
  if (!st->obs || !device_view(c, st->obs, &p, false) || !aligned16(st->obs))
    return bad("storage.obs must be 16-B aligned device memory");
  if ((cfg->tokens > 0) != (st->tokens != nullptr))
    return bad("storage.tokens must be given iff tokens > 0");
  if (st->tokens && (!device_view(c, st->tokens, &p, false) ||
                     !aligned16(st->tokens)))
    return bad("storage.tokens must be 16-B aligned device memory");
  if (tiered) {
    if (!st->host_obs || !device_view(c, st->host_obs, &p, true) ||
        !aligned16(p))
      return bad("storage.host_obs must be page-locked host memory");
    c->st.host_obs = (uint8_t *)p;
    if ((cfg->tokens > 0) != (st->host_tokens != nullptr))
      return bad("storage.host_tokens must be given iff tokens > 0");
    if (st->host_tokens) {
      if (!device_view(c, st->host_tokens, &p, true) || !aligned16(p))
        return bad("storage.host_tokens must be page-locked host memory");
      c->st.host_tokens = (int32_t *)p;
    }
  } else if (st->host_obs || st->host_tokens) {
    return bad("host tier given but hbm_capacity == capacity");
  }
  if (st->action && !device_view(c, st->action, &p, false))
    return bad("storage.action must be device memory");
  if (st->reward && !device_view(c, st->reward, &p, false))
    return bad("storage.reward must be device memory");
  if (st->done && !device_view(c, st->done, &p, false))
    return bad("storage.done must be device memory");

  if (!unit_constants(&c->r1, &c->r2)) return bad("byte/255 self-check failed");
  if (cfg->transform == EDP_XFORM_CHW_NORM_BF16) {
    c->norm_fast = norm_constants(c);
    c->norm_affine = norm_affine_constants(c);
  }

  int dev_sms = 0;
  cudaDeviceGetAttribute(&dev_sms, cudaDevAttrMultiProcessorCount, cfg->device);
  c->coop_sms = dev_sms;

  edp_alloc_fn al = cfg->alloc ? cfg->alloc : default_alloc;
  c->ctrl = (Ctrl *)al(cfg->alloc_user, sizeof(Ctrl));
  if (!c->ctrl) {
    free_all(c);
    delete c;
    return EDP_ERR_OOM;
  }
  Ctrl init{};
  init.max_q = 1u << 20;
  cudaError_t e = cudaMemcpy(c->ctrl, &init, sizeof init, cudaMemcpyHostToDevice);
  if (cfg->prioritized && e == cudaSuccess) {
    uint32_t D = 1;
    uint64_t n = kFanout;
    while (n < c->cap) {
      n *= kFanout;
      ++D;
    }
    c->depth = D;
    c->nleaves = n;
    uint64_t internal = 0, m = 1;
    for (uint32_t d = 0; d < D; ++d) {
      internal += m;
      m *= kFanout;
    }
    const size_t bytes = internal * 8 + n * 4;
    c->tree_mem = al(cfg->alloc_user, bytes);
    c->tree_bytes = bytes;
    if (!c->tree_mem) {
      free_all(c);
      delete c;
      return EDP_ERR_OOM;
    }
    uint64_t off = 0;
    m = 1;
    for (uint32_t d = 0; d < D; ++d) {
      c->level[d] = (uint64_t *)c->tree_mem + off;
      off += m;
      m *= kFanout;
    }
    c->leaves = (uint32_t *)((uint64_t *)c->tree_mem + internal);
    e = cudaMemset(c->tree_mem, 0, bytes);
  }
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) {
    cudaGetLastError();
    free_all(c);
    delete c;
    return EDP_ERR_CUDA;
  }
  *out = c;
  return EDP_OK;
}
#undef bad

edp_status edp_destroy(edp_ctx *ctx) {
  if (!ctx) return EDP_ERR_INVALID;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaDeviceSynchronize();
  free_all(ctx);
  delete ctx;
  return EDP_OK;
}

edp_status edp_migrate(const edp_ctx *src, edp_ctx *dst, edp_stream stream) {
  if (!src || !dst || src == dst) return EDP_ERR_INVALID;
  if (dst->total != 0)
    return fail(dst, EDP_ERR_STATE, "edp_migrate: the destination must be empty");
  const edp_config &a = src->cfg, &b = dst->cfg;
  if (a.transform != b.transform || a.obs_c != b.obs_c || a.obs_h != b.obs_h ||
      a.obs_w != b.obs_w || a.frame_stack != b.frame_stack || a.next_obs != b.next_obs ||
      a.tokens != b.tokens || (a.prioritized != 0) != (b.prioritized != 0) ||
      a.device != b.device)
    return fail(dst, EDP_ERR_STATE,
                "edp_migrate: source and destination differ in layout or device");
  if ((src->st.action != nullptr) != (dst->st.action != nullptr) ||
      (src->st.reward != nullptr) != (dst->st.reward != nullptr) ||
      (src->st.done != nullptr) != (dst->st.done != nullptr))
    return fail(dst, EDP_ERR_STATE, "edp_migrate: metadata arrays differ");
  DeviceGuard dg(b.device);
  EDP_TRACE(__func__);
  cudaStream_t s = (cudaStream_t)stream;
  const uint64_t size = ring_size(src);
  const uint64_t n = size < dst->cap ? size : dst->cap;
  cudaError_t e = launch_migrate(src, dst, src->total - n, n, s);
  if (e == cudaSuccess && dst->depth) {
    // deferred and running-maximum priorities travel with the leaves
    e = cudaMemcpyAsync(&dst->ctrl->pending_q, &src->ctrl->pending_q, 2 * sizeof(uint32_t),
                        cudaMemcpyDeviceToDevice, s);
    if (e == cudaSuccess) e = launch_tree_build_all(dst, s);
  }
  if (e != cudaSuccess) return cuda_fail(dst, e, "edp_migrate");
  dst->total = n;
  return EDP_OK;
}

}  // extern "C"

// ---- checkpoint / resume ------------------------------------------------
namespace {

struct CkptHeader {
  char magic[8];
  uint32_t version, transform, obs_c, obs_h, obs_w, frame_stack, next_obs, tokens;
  uint32_t prioritized, has_action, has_reward, has_done, pending_q, max_q, pad;
  uint64_t n, obs_bytes, tok_bytes;
};
static_assert(sizeof(CkptHeader) == 96, "checkpoint header layout");
constexpr char kMagic[8] = {'E', 'D', 'P', 'C', 'K', 'P', 'T', '1'};
constexpr size_t kStage = 64u << 20;  // bytes staged per transfer

// Where the payload row of logical id L lives (the tier map): the newest
// min(total, cap_h) ids in HBM at L mod cap_h, older ones in the host tier.
uint8_t *row_of(const edp_ctx *c, uint8_t *hbm, uint8_t *host, uint64_t row, uint64_t L) {
  const uint64_t in_hbm = c->total < c->cap_h ? c->total : c->cap_h;
  if (L >= c->total - in_hbm) return hbm + (L % c->cap_h) * row;
  return host + (L % (c->cap_c ? c->cap_c : 1)) * row;
}

// Visit ids [L0, L0 + n) in order as runs of consecutive rows of one array:
// fn(first id, count, pointer to the first row).
template <typename F>
void payload_runs(const edp_ctx *c, uint8_t *hbm, uint8_t *host, uint64_t row, uint64_t L0,
                  uint64_t n, F fn) {
  uint64_t j = 0;
  while (j < n) {
    uint8_t *p = row_of(c, hbm, host, row, L0 + j);
    uint64_t k = 1;
    while (j + k < n && row_of(c, hbm, host, row, L0 + j + k) == p + k * row) ++k;
    fn(j, k, p);
    j += k;
  }
}

// The same for an array indexed by slot L mod cap.
template <typename F>
void slot_runs(uint64_t cap, uint64_t L0, uint64_t n, F fn) {
  uint64_t j = 0;
  while (j < n) {
    const uint64_t s = (L0 + j) % cap;
    const uint64_t k = std::min<uint64_t>(n - j, cap - s);
    fn(j, k, s);
    j += k;
  }
}

// Bytes a checkpoint of n transitions with header h occupies: the header,
// then per transition its payload rows and the metadata arrays it carries.
// False when the count cannot be a real checkpoint's (the product would
// overflow).
bool ckpt_bytes(const CkptHeader &h, uint64_t *out) {
  const uint64_t per = h.obs_bytes + h.tok_bytes + 4u * (h.has_action != 0) +
                       4u * (h.has_reward != 0) + 1u * (h.has_done != 0) +
                       4u * (h.prioritized != 0);
  if (h.n > (UINT64_MAX - sizeof(CkptHeader)) / (per ? per : 1)) return false;
  *out = sizeof(CkptHeader) + h.n * per;
  return true;
}

bool same_layout(const edp_ctx *c, const CkptHeader &h) {
  const edp_config &g = c->cfg;
  return h.transform == g.transform && h.obs_c == g.obs_c && h.obs_h == g.obs_h &&
         h.obs_w == g.obs_w && h.frame_stack == g.frame_stack && h.next_obs == g.next_obs &&
         h.tokens == g.tokens && h.prioritized == (g.prioritized != 0) &&
         h.has_action == (c->st.action != nullptr) && h.has_reward == (c->st.reward != nullptr) &&
         h.has_done == (c->st.done != nullptr);
}

}  // namespace

extern "C" {

edp_status edp_save(edp_ctx *ctx, const char *path, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!path) return fail(ctx, EDP_ERR_INVALID, "edp_save: path is NULL");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_save");
  CkptHeader h{};
  std::memcpy(h.magic, kMagic, 8);
  h.version = 1;
  const edp_config &g = ctx->cfg;
  h.transform = g.transform; h.obs_c = g.obs_c; h.obs_h = g.obs_h; h.obs_w = g.obs_w;
  h.frame_stack = g.frame_stack; h.next_obs = g.next_obs; h.tokens = g.tokens;
  h.prioritized = g.prioritized != 0;
  h.has_action = ctx->st.action != nullptr;
  h.has_reward = ctx->st.reward != nullptr;
  h.has_done = ctx->st.done != nullptr;
  h.n = ring_size(ctx);
  h.obs_bytes = ctx->obs_bytes;
  h.tok_bytes = ctx->tok_bytes;
  if (ctx->depth) {
    uint32_t pm[2];
    e = cudaMemcpy(pm, &ctx->ctrl->pending_q, sizeof pm, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_save");
    h.pending_q = pm[0];
    h.max_q = pm[1];
  }
  FILE *f = std::fopen(path, "wb");
  if (!f) return fail(ctx, EDP_ERR_INVALID, "edp_save: cannot open %s", path);
  uint8_t *stage = (uint8_t *)std::malloc(kStage);
  const bool staged = stage != nullptr;
  bool ok = staged && std::fwrite(&h, sizeof h, 1, f) == 1;
  const uint64_t L0 = ctx->total - h.n;
  // copy `bytes` from (device or host) src to the file through the stage
  auto put = [&](const void *src, uint64_t bytes) {
    for (uint64_t o = 0; ok && o < bytes; o += kStage) {
      const size_t b = (size_t)std::min<uint64_t>(kStage, bytes - o);
      ok = cudaMemcpy(stage, (const uint8_t *)src + o, b, cudaMemcpyDefault) == cudaSuccess &&
           std::fwrite(stage, 1, b, f) == b;
    }
  };
  auto payload = [&](uint8_t *hbm, uint8_t *host, uint64_t row) {
    payload_runs(ctx, hbm, host, row, L0, h.n,
                 [&](uint64_t, uint64_t k, uint8_t *p) { put(p, k * row); });
  };
  payload(ctx->st.obs, ctx->st.host_obs, ctx->obs_bytes);
  if (ctx->tok_bytes)
    payload((uint8_t *)ctx->st.tokens, (uint8_t *)ctx->st.host_tokens, ctx->tok_bytes);
  auto meta = [&](const void *base, size_t elem) {
    if (!base) return;
    slot_runs(ctx->cap, L0, h.n, [&](uint64_t, uint64_t k, uint64_t sl) {
      put((const uint8_t *)base + sl * elem, k * elem);
    });
  };
  meta(ctx->st.action, 4);
  meta(ctx->st.reward, 4);
  meta(ctx->st.done, 1);
  meta(ctx->leaves, 4);
  std::free(stage);
  ok = (std::fclose(f) == 0) && ok;
  if (!ok) {
    cudaGetLastError();
    return fail(ctx, staged ? EDP_ERR_INVALID : EDP_ERR_OOM, "edp_save: writing %s failed",
                path);
  }
  return EDP_OK;
}

edp_status edp_load(edp_ctx *ctx, const char *path, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!path) return fail(ctx, EDP_ERR_INVALID, "edp_load: path is NULL");
  if (ctx->total != 0) return fail(ctx, EDP_ERR_STATE, "edp_load: the context must be empty");
  FILE *f = std::fopen(path, "rb");
  if (!f) return fail(ctx, EDP_ERR_INVALID, "edp_load: cannot open %s", path);
  CkptHeader h{};
  if (std::fread(&h, sizeof h, 1, f) != 1 || std::memcmp(h.magic, kMagic, 8) != 0 ||
      h.version != 1) {
    std::fclose(f);
    return fail(ctx, EDP_ERR_INVALID, "edp_load: %s is not a checkpoint of this format", path);
  }
  if (!same_layout(ctx, h) || h.obs_bytes != ctx->obs_bytes || h.tok_bytes != ctx->tok_bytes) {
    std::fclose(f);
    return fail(ctx, EDP_ERR_STATE, "edp_load: the checkpoint's layout differs from the context's");
  }
  // a truncated or padded file is refused before anything is written
  uint64_t want = 0;
  long have = -1;
  if (std::fseek(f, 0, SEEK_END) == 0) have = std::ftell(f);
  if (!ckpt_bytes(h, &want) || have < 0 || (uint64_t)have != want ||
      std::fseek(f, (long)sizeof h, SEEK_SET) != 0) {
    std::fclose(f);
    return fail(ctx, EDP_ERR_INVALID,
                "edp_load: %s holds %ld bytes, its header describes %llu (truncated file?)", path,
                have, (unsigned long long)want);
  }
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  const uint64_t n = h.n < ctx->cap ? h.n : ctx->cap;  // the newest n are kept
  const uint64_t skip = h.n - n;
  uint8_t *stage = (uint8_t *)std::malloc(kStage);
  const bool staged = stage != nullptr;
  bool ok = staged;
  // the context's cursors as they will be: n insertions, ids 0 .. n-1
  ctx->total = n;
  auto get = [&](void *dst, uint64_t bytes) {
    for (uint64_t o = 0; ok && o < bytes; o += kStage) {
      const size_t b = (size_t)std::min<uint64_t>(kStage, bytes - o);
      ok = std::fread(stage, 1, b, f) == b &&
           cudaMemcpy((uint8_t *)dst + o, stage, b, cudaMemcpyDefault) == cudaSuccess;
    }
  };
  auto seek = [&](uint64_t bytes) {
    if (ok && bytes) ok = std::fseek(f, (long)bytes, SEEK_CUR) == 0;
  };
  auto payload = [&](uint8_t *hbm, uint8_t *host, uint64_t row) {
    seek(skip * row);
    payload_runs(ctx, hbm, host, row, 0, n,
                 [&](uint64_t, uint64_t k, uint8_t *p) { get(p, k * row); });
  };
  payload(ctx->st.obs, ctx->st.host_obs, ctx->obs_bytes);
  if (ctx->tok_bytes)
    payload((uint8_t *)ctx->st.tokens, (uint8_t *)ctx->st.host_tokens, ctx->tok_bytes);
  auto meta = [&](void *base, size_t elem, bool present) {
    if (!present) return;
    seek(skip * elem);
    slot_runs(ctx->cap, 0, n, [&](uint64_t, uint64_t k, uint64_t sl) {
      get((uint8_t *)base + sl * elem, k * elem);
    });
  };
  meta(ctx->st.action, 4, h.has_action);
  meta(ctx->st.reward, 4, h.has_reward);
  meta(ctx->st.done, 1, h.has_done);
  meta(ctx->leaves, 4, h.prioritized);
  std::free(stage);
  std::fclose(f);
  cudaError_t e = cudaSuccess;
  if (ok && ctx->depth) {
    const uint32_t pm[2] = {h.pending_q, h.max_q};
    e = cudaMemcpy(&ctx->ctrl->pending_q, pm, sizeof pm, cudaMemcpyHostToDevice);
    if (e == cudaSuccess) e = launch_tree_build_all(ctx, (cudaStream_t)stream);
  }
  if (!ok || e != cudaSuccess) {
    // back to an empty context: no transition, and no leaf or sum left over
    // from the rows read before the failure
    ctx->total = 0;
    cudaGetLastError();
    if (ctx->depth) {
      const uint32_t pm[2] = {0, 1u << 20};
      cudaStreamSynchronize((cudaStream_t)stream);
      cudaMemset(ctx->tree_mem, 0, ctx->tree_bytes);
      cudaMemcpy(&ctx->ctrl->pending_q, pm, sizeof pm, cudaMemcpyHostToDevice);
      cudaGetLastError();
    }
    return fail(ctx, staged ? EDP_ERR_INVALID : EDP_ERR_OOM, "edp_load: reading %s failed",
                path);
  }
  return EDP_OK;
}

edp_status edp_get_info(const edp_ctx *ctx, edp_info *o) {
  if (!ctx || !o) return EDP_ERR_INVALID;
  memset(o, 0, sizeof *o);
  o->capacity = ctx->cap;
  o->hbm_capacity = ctx->cap_h;
  o->total = ctx->total;
  o->size = ring_size(ctx);
  o->head = ctx->total % ctx->cap;
  o->oldest = (ctx->total - o->size) % ctx->cap;
  o->n_valid = n_valid(ctx);
  o->tree_depth = ctx->depth;
  if (ctx->cfg.transform == EDP_XFORM_CHW_NORM_BF16)
    o->norm_path = ctx->norm_affine ? 2 : ctx->norm_fast ? 1 : 0;
  o->tree_fanout = kFanout;
  o->tree_leaves = ctx->leaves;
  for (uint32_t d = 0; d < ctx->depth && d < 8; ++d) o->tree_level[d] = ctx->level[d];
  o->pending_q = &ctx->ctrl->pending_q;
  o->max_q = &ctx->ctrl->max_q;
  return EDP_OK;
}

edp_status edp_ingest(edp_ctx *ctx, const edp_fields *src, uint64_t n,
                      const uint32_t *q, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!src) return fail(ctx, EDP_ERR_INVALID, "edp_ingest: src is NULL");
  if (n > ctx->cap)
    return fail(ctx, EDP_ERR_INVALID, "edp_ingest: n=%llu exceeds capacity",
                (unsigned long long)n);
  if (n == 0) return EDP_OK;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaStream_t s = (cudaStream_t)stream;
  edp_fields f{};
  const void *p;
  if (!src->obs || !device_view(ctx, src->obs, &p, true) || !aligned16(p))
    return fail(ctx, EDP_ERR_INVALID,
                "edp_ingest: src.obs must be 16-B aligned device or page-locked memory");
  f.obs = (const uint8_t *)p;
  if ((ctx->tok_bytes > 0) != (src->tokens != nullptr))
    return fail(ctx, EDP_ERR_INVALID, "edp_ingest: src.tokens given iff tokens > 0");
  if (src->tokens) {
    if (!device_view(ctx, src->tokens, &p, true) || !aligned16(p))
      return fail(ctx, EDP_ERR_INVALID, "edp_ingest: bad src.tokens");
    f.tokens = (const int32_t *)p;
  }
#define EDP_VIEW(field, T)                                                     \
  if (src->field) {                                                            \
    if (!device_view(ctx, src->field, &p, true))                               \
      return fail(ctx, EDP_ERR_INVALID, "edp_ingest: bad src." #field);        \
    f.field = (T)p;                                                            \
  }
  EDP_VIEW(action, const int32_t *)
  EDP_VIEW(reward, const float *)
  EDP_VIEW(done, const uint8_t *)
#undef EDP_VIEW
  if (q && !device_view(ctx, q, &p, false))
    return fail(ctx, EDP_ERR_INVALID, "edp_ingest: q must be device memory");
  if (q && !ctx->depth)
    return fail(ctx, EDP_ERR_STATE, "edp_ingest: q given to a context without priorities");

  cudaError_t e = cudaSuccess;
  // Placement of ids [T, T+n).  Afterwards HBM holds [Tn - keep_h, Tn) and
  // the host tier [Tn - keep, Tn - keep_h).  Resident ids that leave HBM
  // but stay retained are demoted first (same stream, so before their HBM
  // slots are overwritten); new ids older than the HBM window go straight
  // to the host tier; the rest are written to HBM.
  const uint64_t T = ctx->total, Tn = T + n;
  const uint64_t keep_h = Tn < ctx->cap_h ? Tn : ctx->cap_h;
  const uint64_t keep = Tn < ctx->cap ? Tn : ctx->cap;
  uint64_t new_hbm_lo = T;
  bool swapped = false;
  uint64_t demoted = 0, to_host = 0;  // rows moved into the host tier
  if (ctx->cap_c) {
    const uint64_t in_hbm = T < ctx->cap_h ? T : ctx->cap_h;
    uint64_t lo = T - in_hbm;
    if (lo < Tn - keep) lo = Tn - keep;  // evicted outright
    const uint64_t hi = (Tn - keep_h) < T ? (Tn - keep_h) : T;
    // new ids [max(T, Tn - keep), Tn - keep_h) -> host tier directly
    const uint64_t dlo = T > Tn - keep ? T : Tn - keep;
    const uint64_t dhi = Tn - keep_h;
    if (new_hbm_lo < Tn - keep_h) new_hbm_lo = Tn - keep_h;
    // steady state: every new id takes the HBM slot of the id it demotes
    // (id L leaves, id L + cap_h arrives) -> one fused pass, both link
    // directions at once
    swapped = hi > lo && dhi <= dlo && hi - lo == Tn - new_hbm_lo &&
              lo + ctx->cap_h == new_hbm_lo;
    demoted = hi > lo ? hi - lo : 0;
    to_host = dhi > dlo ? dhi - dlo : 0;
    if (swapped) {
      const uint64_t skip = new_hbm_lo - T;
      e = launch_swap(ctx, lo, f.obs + skip * ctx->obs_bytes,
                      f.tokens ? f.tokens + skip * (ctx->tok_bytes / 4) : nullptr,
                      hi - lo, s);
    } else {
      if (hi > lo) e = launch_demote(ctx, lo, hi - lo, s);
      if (e == cudaSuccess && dhi > dlo)
        e = launch_copy_rows_to_host(ctx, f.obs, f.tokens, dlo - T, dlo, dhi - dlo, s);
    }
    if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_ingest(host tier)");
  }
  // leaves whose tree sums change: the new ones and, with next_obs, the
  // previous newest (its deferred priority lands now)
  uint64_t tfirst = ctx->total % ctx->cap, tcount = n;
  if (ctx->defer && ctx->total >= 1) {
    tfirst = (ctx->total - 1) % ctx->cap;
    tcount = n + 1;
  }
  if (tcount > ctx->cap) tcount = ctx->cap;
  // traffic: source rows and metadata read; ring rows written to their
  // tier (demoted rows read from HBM and written to the host); metadata
  // and leaves written to HBM
  auto count_ingest = [&]() {
    const uint64_t R = ctx->obs_bytes + ctx->tok_bytes;
    count_read(ctx, src->obs, n * ctx->obs_bytes);
    count_read(ctx, src->tokens, n * ctx->tok_bytes);
    count_read(ctx, src->action, 4 * n);
    count_read(ctx, src->reward, 4 * n);
    count_read(ctx, src->done, n);
    count_read(ctx, q, 4 * n);
    ctx->cnt.hbm_write += (n - to_host) * R;
    ctx->cnt.link_write += (to_host + demoted) * R;
    ctx->cnt.hbm_read += demoted * R;
    ctx->cnt.hbm_write += n * (4 * (ctx->st.action != nullptr) + 4 * (ctx->st.reward != nullptr) +
                               (ctx->st.done != nullptr) + 4 * (ctx->leaves != nullptr));
    ctx->cnt.ingested += n;
    ++ctx->cnt.calls;
  };
  if (e == cudaSuccess && ingest_fusable(ctx, n)) {
    // single tier, a moderate n: the whole insertion in one launch
    e = launch_ingest_fused(ctx, &f, n, q, tfirst, ctx->depth ? tcount : 0, s);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_ingest");
    count_ingest();
    ctx->total += n;
    return EDP_OK;
  }
  // metadata and leaves, then the tree above them, then the payload rows:
  // the row copy starts behind the (waiting) metadata and tree kernels and
  // overlaps the last of them, since neither reads the rows
  const bool meta = ctx->st.action || ctx->st.reward || ctx->st.done || ctx->leaves;
  if (e == cudaSuccess) e = launch_ingest_meta(ctx, &f, n, q, s);
  if (e == cudaSuccess && ctx->depth) e = launch_tree_refresh(ctx, tfirst, tcount, s);
  const uint64_t skip = new_hbm_lo - T, nh = Tn - new_hbm_lo;
  if (e == cudaSuccess && !swapped) {
    e = launch_copy_rows(ctx->st.obs, ctx->cap_h, new_hbm_lo % ctx->cap_h,
                         f.obs + skip * ctx->obs_bytes, nh, ctx->obs_bytes, s, !meta);
    if (e == cudaSuccess && ctx->tok_bytes)
      e = launch_copy_rows((uint8_t *)ctx->st.tokens, ctx->cap_h,
                           new_hbm_lo % ctx->cap_h,
                           (const uint8_t *)f.tokens + skip * ctx->tok_bytes, nh,
                           ctx->tok_bytes, s, false);  // behind the row copy
  }
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_ingest");
  count_ingest();
  ctx->total += n;
  return EDP_OK;
}

edp_status edp_sample(edp_ctx *ctx, edp_sample_mode mode, uint32_t batch,
                      uint64_t seed, uint64_t round, int64_t *idx, uint32_t *q,
                      edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!idx) return fail(ctx, EDP_ERR_INVALID, "edp_sample: idx is NULL");
  if (batch == 0) return fail(ctx, EDP_ERR_INVALID, "edp_sample: batch == 0");
  const void *p;
  if (!device_view(ctx, idx, &p, false) || (q && !device_view(ctx, q, &p, false)))
    return fail(ctx, EDP_ERR_INVALID, "edp_sample: outputs must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaStream_t s = (cudaStream_t)stream;
  cudaError_t e;
  switch (mode) {
    case EDP_SAMPLE_UNIFORM:
      if (n_valid(ctx) == 0)
        return fail(ctx, EDP_ERR_EMPTY, "edp_sample: no sampleable transition");
      e = launch_sample_uniform(ctx, batch, seed, round, idx, s);
      break;
    case EDP_SAMPLE_PRIORITIZED:
      if (!ctx->depth)
        return fail(ctx, EDP_ERR_STATE, "edp_sample: context has no priorities");
      if (n_valid(ctx) == 0)
        return fail(ctx, EDP_ERR_EMPTY, "edp_sample: no sampleable transition");
      e = launch_sample_prioritized(ctx, batch, seed, round, idx, q, s);
      break;
    case EDP_SAMPLE_PERMUTE:
      if (ring_size(ctx) == 0)
        return fail(ctx, EDP_ERR_EMPTY, "edp_sample: ring is empty");
      if (batch != ring_size(ctx))
        return fail(ctx, EDP_ERR_INVALID,
                    "edp_sample: PERMUTE needs batch == size (%llu)",
                    (unsigned long long)ring_size(ctx));
      e = launch_permute(ctx, batch, seed, round, idx, s);
      break;
    default:
      return fail(ctx, EDP_ERR_INVALID, "edp_sample: unknown mode %d", (int)mode);
  }
  if (e != cudaSuccess) return launch_fail(ctx, e, "edp_sample");
  count_hbm(ctx, 0, 8ull * batch + (q && mode == EDP_SAMPLE_PRIORITIZED ? 4ull * batch : 0));
  ctx->cnt.sampled += batch;
  return EDP_OK;
}

// Argument checks shared by edp_deliver and edp_sample_deliver; *res is
// the batch with every output resolved to a device-usable address (an
// output may be page-locked host memory: the kernel then writes it over the
// host link).
static edp_status deliver_checks(edp_ctx *ctx, const int64_t *idx, uint32_t batch,
                                 const edp_batch *out, edp_batch *res) {
  if (!idx || !out || !out->obs)
    return fail(ctx, EDP_ERR_INVALID, "edp_deliver: idx/out/out->obs is NULL");
  if (batch == 0) return fail(ctx, EDP_ERR_INVALID, "edp_deliver: batch == 0");
  if (ring_size(ctx) == 0) return fail(ctx, EDP_ERR_EMPTY, "edp_deliver: ring is empty");
  if (out->next_obs && !ctx->defer)
    return fail(ctx, EDP_ERR_STATE, "edp_deliver: next_obs needs next_obs=1");
  if (out->tokens && !ctx->tok_bytes)
    return fail(ctx, EDP_ERR_STATE, "edp_deliver: context stores no tokens");
  if (out->action && !ctx->st.action)
    return fail(ctx, EDP_ERR_STATE, "edp_deliver: context stores no action");
  if (out->reward && !ctx->st.reward)
    return fail(ctx, EDP_ERR_STATE, "edp_deliver: context stores no reward");
  if (out->done && !ctx->st.done)
    return fail(ctx, EDP_ERR_STATE, "edp_deliver: context stores no done");
  if (out->isw && !out->q)
    return fail(ctx, EDP_ERR_INVALID, "edp_deliver: isw needs q");
  if (out->isw && !(out->beta >= 0.0))
    return fail(ctx, EDP_ERR_INVALID, "edp_deliver: beta must be >= 0");
  for (int i = 0; i < 2; ++i)
    if ((out->gather_src[i] == nullptr) != (out->gather_dst[i] == nullptr))
      return fail(ctx, EDP_ERR_INVALID, "edp_deliver: gather pair %d half-NULL", i);
  const void *p;
  const void *ins[] = {idx, out->q, out->gather_src[0], out->gather_src[1]};
  for (const void *o : ins)
    if (o && !device_view(ctx, o, &p, false))
      return fail(ctx, EDP_ERR_INVALID, "edp_deliver: inputs must be device memory");
  *res = *out;
  void **outs[] = {&res->obs, &res->next_obs, reinterpret_cast<void **>(&res->action),
                   reinterpret_cast<void **>(&res->reward),
                   reinterpret_cast<void **>(&res->done),
                   reinterpret_cast<void **>(&res->tokens),
                   reinterpret_cast<void **>(&res->isw),
                   reinterpret_cast<void **>(&res->gather_dst[0]),
                   reinterpret_cast<void **>(&res->gather_dst[1])};
  for (void **o : outs) {
    if (!*o) continue;
    if (!device_view(ctx, *o, &p, true))
      return fail(ctx, EDP_ERR_INVALID,
                  "edp_deliver: outputs must be device or page-locked host memory");
    *o = const_cast<void *>(p);
  }
  if (!aligned16(res->obs) || (res->next_obs && !aligned16(res->next_obs)) ||
      (res->tokens && !aligned16(res->tokens)))
    return fail(ctx, EDP_ERR_INVALID, "edp_deliver: obs/next_obs/tokens 16-B aligned");
  return EDP_OK;
}

// Traffic of a delivery of B entries into `out` (the caller's pointers):
// per entry the unique source bytes (the K or K + 1 frames of a stack, the
// image and tokens otherwise) and the scalars read, and every output
// written to its memory.  A two-tier ring's host rows are counted on the
// device and moved to link_read by edp_get_counters.
static void count_deliver(edp_ctx *ctx, uint32_t B, const edp_batch *out) {
  const auto &cfg = ctx->cfg;
  const uint64_t F = ctx->obs_bytes;
  uint64_t per = F, obs_out = 0;
  if (cfg.transform == EDP_XFORM_STACK_F32) {
    per = F * (cfg.frame_stack + (out->next_obs ? 1 : 0));
    obs_out = F * cfg.frame_stack * 4;
  } else {
    per = F + (out->tokens ? ctx->tok_bytes : 0);
    obs_out = F * 2;
  }
  const uint64_t scalars = 8 + 4 * (out->action != nullptr) + 4 * (out->reward != nullptr) +
                           (out->done != nullptr) + 4 * (out->q != nullptr) +
                           4 * (out->gather_src[0] != nullptr) + 4 * (out->gather_src[1] != nullptr);
  ctx->cnt.hbm_read += B * (per + scalars);
  count_write(ctx, out->obs, B * obs_out);
  count_write(ctx, out->next_obs, B * obs_out);
  count_write(ctx, out->tokens, B * ctx->tok_bytes);
  count_write(ctx, out->action, 4ull * B);
  count_write(ctx, out->reward, 4ull * B);
  count_write(ctx, out->done, 1ull * B);
  count_write(ctx, out->isw, 4ull * B);
  count_write(ctx, out->gather_dst[0], 4ull * B);
  count_write(ctx, out->gather_dst[1], 4ull * B);
  ctx->cnt.delivered += B;
  ++ctx->cnt.calls;
}

edp_status edp_deliver(edp_ctx *ctx, const int64_t *idx, uint32_t batch,
                       const edp_batch *out, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  edp_batch res;
  const edp_status st = deliver_checks(ctx, idx, batch, out, &res);
  if (st != EDP_OK) return st;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_deliver(ctx, idx, batch, &res, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_deliver");
  count_deliver(ctx, batch, out);
  return EDP_OK;
}

edp_status edp_sample_deliver(edp_ctx *ctx, uint32_t batch, uint64_t seed, uint64_t round,
                              int64_t *idx, const edp_batch *out, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (n_valid(ctx) == 0)
    return fail(ctx, EDP_ERR_EMPTY, "edp_sample_deliver: no sampleable transition");
  if (out && (out->isw || out->q))
    return fail(ctx, EDP_ERR_INVALID,
                "edp_sample_deliver: uniform draws carry no priorities (q/isw must be NULL)");
  edp_batch res;
  const edp_status st = deliver_checks(ctx, idx, batch, out, &res);
  if (st != EDP_OK) return st;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  DrawUniform d{seed, round, idx};
  cudaError_t e = launch_deliver(ctx, idx, batch, &res, (cudaStream_t)stream, &d);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_sample_deliver");
  count_deliver(ctx, batch, out);  // the drawn indices are written, not read:
  ctx->cnt.hbm_read -= 8ull * batch;  // the index bytes count once, as a write
  ctx->cnt.hbm_write += 8ull * batch;
  ctx->cnt.sampled += batch;
  return EDP_OK;
}

static edp_status update_common(edp_ctx *ctx, const char *who, const int64_t *idx,
                                const uint32_t *q, const float *td, uint32_t n,
                                double alpha, double eps, edp_stream stream) {
  const edp_status st = update_args(ctx, who, idx, q, td, n, alpha, eps);
  if (st != EDP_OK || n == 0) return st;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(who);
  cudaError_t e = launch_update(ctx, idx, q, td, alpha, eps, n, (cudaStream_t)stream);
  if (e != cudaSuccess) return launch_fail(ctx, e, who);
  count_hbm(ctx, 12ull * n, 4ull * n);  // pairs read, leaves written
  return EDP_OK;
}

edp_status edp_update_priorities(edp_ctx *ctx, const int64_t *idx,
                                 const uint32_t *q, uint32_t n,
                                 edp_stream stream) {
  if (ctx && n && !q) return fail(ctx, EDP_ERR_INVALID, "edp_update_priorities: q NULL");
  return update_common(ctx, "edp_update_priorities", idx, q, nullptr, n, 0.0, 0.0, stream);
}

edp_status edp_update_priorities_td(edp_ctx *ctx, const int64_t *idx,
                                    const float *td, uint32_t n, double alpha,
                                    double eps, edp_stream stream) {
  if (ctx && n && !td) return fail(ctx, EDP_ERR_INVALID, "edp_update_priorities_td: td NULL");
  return update_common(ctx, "edp_update_priorities_td", idx, nullptr, td, n, alpha, eps,
                       stream);
}

edp_status edp_priorities_from_td(edp_ctx *ctx, const float *td, uint32_t n,
                                  double alpha, double eps, uint32_t *q,
                                  edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (n == 0) return EDP_OK;
  const void *p;
  if (!td || !q || !device_view(ctx, td, &p, false) || !device_view(ctx, q, &p, false))
    return fail(ctx, EDP_ERR_INVALID, "edp_priorities_from_td: device arrays required");
  if (!(alpha >= 0.0 && eps >= 0.0))
    return fail(ctx, EDP_ERR_INVALID, "edp_priorities_from_td: alpha, eps >= 0");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_prio_from_td(td, n, alpha, eps, q, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_priorities_from_td");
  count_hbm(ctx, 4ull * n, 4ull * n);
  return EDP_OK;
}

edp_status edp_gae(edp_ctx *ctx, const float *r, const float *v,
                   const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                   double lambda, float *adv, float *ret, float *adv_norm,
                   edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!r || !v || !d) return fail(ctx, EDP_ERR_INVALID, "edp_gae: r/v/d NULL");
  if (T == 0 || E == 0 || (uint64_t)T * E > 0x7FFFFFFFull)
    return fail(ctx, EDP_ERR_INVALID, "edp_gae: need T, E >= 1 and T*E < 2^31");
  if (!std::isfinite(gamma) || !std::isfinite(lambda))
    return fail(ctx, EDP_ERR_INVALID, "edp_gae: gamma/lambda not finite");
  const void *p;
  const void *ptrs[] = {r, v, d, adv, ret, adv_norm};
  for (const void *o : ptrs)
    if (o && !device_view(ctx, o, &p, false))
      return fail(ctx, EDP_ERR_INVALID, "edp_gae: arrays must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_gae(ctx, r, v, d, T, E, gamma, lambda, adv, ret, adv_norm,
                             (cudaStream_t)stream);
  if (e != cudaSuccess) return launch_fail(ctx, e, "edp_gae");
  const uint64_t te = (uint64_t)T * E;
  count_hbm(ctx, 9 * te + 4ull * E,
            4 * te * ((adv != nullptr) + (ret != nullptr) + (adv_norm != nullptr)));
  return EDP_OK;
}

// ---- sharded buffer -------------------------------------------------------

// true when every non-NULL pointer is device memory of the context's GPU
static bool all_device(const edp_ctx *ctx, std::initializer_list<const void *> ps) {
  const void *p;
  for (const void *o : ps)
    if (o && !device_view(ctx, o, &p, false)) return false;
  return true;
}

edp_status edp_tree_total(edp_ctx *ctx, uint64_t *d_total, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!ctx->depth) return fail(ctx, EDP_ERR_STATE, "edp_tree_total: context has no priorities");
  if (!d_total || !all_device(ctx, {d_total}))
    return fail(ctx, EDP_ERR_INVALID, "edp_tree_total: d_total must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_tree_total(ctx, d_total, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_tree_total");
  count_hbm(ctx, 8, 8);
  return EDP_OK;
}

edp_status edp_route_prioritized(edp_ctx *ctx, const uint64_t *d_totals, uint32_t G,
                                 uint32_t batch, uint32_t k0, uint32_t n, uint64_t seed,
                                 uint64_t round, uint64_t *d_local_t, int64_t *d_counts,
                                 edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (G == 0 || G > 1024)
    return fail(ctx, EDP_ERR_INVALID, "edp_route_prioritized: G must be in [1, 1024]");
  if (batch == 0) return fail(ctx, EDP_ERR_INVALID, "edp_route_prioritized: batch == 0");
  if ((uint64_t)k0 + n > batch)
    return fail(ctx, EDP_ERR_INVALID, "edp_route_prioritized: k0 + n > batch");
  if (!d_totals || !d_counts || (n && !d_local_t) ||
      !all_device(ctx, {d_totals, d_counts, d_local_t}))
    return fail(ctx, EDP_ERR_INVALID,
                "edp_route_prioritized: totals, local targets and counts must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_route_prioritized(ctx, d_totals, G, batch, k0, n, seed, round,
                                           d_local_t, d_counts, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_route_prioritized");
  count_hbm(ctx, 8ull * G, 8ull * n + 8ull * G);
  return EDP_OK;
}

edp_status edp_sample_targets(edp_ctx *ctx, const uint64_t *d_targets, uint32_t n,
                              int64_t *d_idx, uint32_t *d_q, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!ctx->depth)
    return fail(ctx, EDP_ERR_STATE, "edp_sample_targets: context has no priorities");
  if (n == 0) return EDP_OK;
  if (!d_targets || !d_idx || !all_device(ctx, {d_targets, d_idx, d_q}))
    return fail(ctx, EDP_ERR_INVALID,
                "edp_sample_targets: targets, idx and q must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_sample_targets(ctx, d_targets, n, d_idx, d_q, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_sample_targets");
  count_hbm(ctx, 8ull * n, (d_q ? 12ull : 8ull) * n);
  ctx->cnt.sampled += n;
  return EDP_OK;
}

edp_status edp_batch_qmin(edp_ctx *ctx, const uint32_t *d_q, uint32_t n, int64_t *d_qmin,
                          edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!d_qmin || (n && !d_q) || !all_device(ctx, {d_q, d_qmin}))
    return fail(ctx, EDP_ERR_INVALID, "edp_batch_qmin: q and qmin must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_batch_qmin(ctx, d_q, n, d_qmin, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_batch_qmin");
  count_hbm(ctx, 4ull * n, 8);
  return EDP_OK;
}

edp_status edp_is_weights(edp_ctx *ctx, const uint32_t *d_q, uint32_t n,
                          const int64_t *d_qmin, double beta, float *d_w, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!(beta >= 0.0)) return fail(ctx, EDP_ERR_INVALID, "edp_is_weights: beta must be >= 0");
  if (n == 0) return EDP_OK;
  if (!d_q || !d_qmin || !d_w || !all_device(ctx, {d_q, d_qmin, d_w}))
    return fail(ctx, EDP_ERR_INVALID, "edp_is_weights: q, qmin and w must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_is_weights(ctx, d_q, n, d_qmin, beta, d_w, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_is_weights");
  count_hbm(ctx, 4ull * n + 8, 4ull * n);
  return EDP_OK;
}

edp_status edp_gae_stats(edp_ctx *ctx, const float *r, const float *v, const uint8_t *d,
                         uint32_t T, uint32_t E, double gamma, double lambda, float *adv,
                         float *ret, double *d_stats, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!r || !v || !d) return fail(ctx, EDP_ERR_INVALID, "edp_gae_stats: r/v/d NULL");
  if (!adv || !d_stats) return fail(ctx, EDP_ERR_INVALID, "edp_gae_stats: adv/stats NULL");
  if (T == 0 || E == 0 || (uint64_t)T * E > 0x7FFFFFFFull)
    return fail(ctx, EDP_ERR_INVALID, "edp_gae_stats: need T, E >= 1 and T*E < 2^31");
  if (!std::isfinite(gamma) || !std::isfinite(lambda))
    return fail(ctx, EDP_ERR_INVALID, "edp_gae_stats: gamma/lambda not finite");
  if (!all_device(ctx, {r, v, d, adv, ret, d_stats}))
    return fail(ctx, EDP_ERR_INVALID, "edp_gae_stats: arrays must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_gae_stats(ctx, r, v, d, T, E, gamma, lambda, adv, ret, d_stats,
                                   (cudaStream_t)stream);
  if (e != cudaSuccess) return launch_fail(ctx, e, "edp_gae_stats");
  const uint64_t te = (uint64_t)T * E;
  count_hbm(ctx, 9 * te + 4ull * E, 4 * te * (1 + (ret != nullptr)) + 24);
  return EDP_OK;
}

edp_status edp_gae_normalize(edp_ctx *ctx, const float *adv, uint64_t n, const double *d_stats,
                             float *adv_norm, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (n == 0 || n > 0x7FFFFFFFull)
    return fail(ctx, EDP_ERR_INVALID, "edp_gae_normalize: need 1 <= n < 2^31");
  if (!adv || !d_stats || !adv_norm || !all_device(ctx, {adv, d_stats, adv_norm}))
    return fail(ctx, EDP_ERR_INVALID, "edp_gae_normalize: arrays must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_gae_normalize(ctx, adv, n, d_stats, adv_norm, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_gae_normalize");
  count_hbm(ctx, 4 * n + 24, 4 * n);
  return EDP_OK;
}

edp_status edp_grpo_advantage(edp_ctx *ctx, const float *r, const uint64_t *group_off,
                              uint32_t n_groups, float eps, float *adv, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!r || !group_off || !adv || n_groups == 0)
    return fail(ctx, EDP_ERR_INVALID, "edp_grpo_advantage: NULL array or no group");
  if (!(eps >= 0.f) || !std::isfinite(eps))
    return fail(ctx, EDP_ERR_INVALID, "edp_grpo_advantage: eps must be finite and >= 0");
  const void *p;
  const void *ptrs[] = {r, group_off, adv};
  for (const void *o : ptrs)
    if (!device_view(ctx, o, &p, false))
      return fail(ctx, EDP_ERR_INVALID, "edp_grpo_advantage: arrays must be device memory");
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_grpo(ctx, r, group_off, n_groups, eps, adv, (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_grpo_advantage");
  count_hbm(ctx, 8ull * (n_groups + 1), 0);  // the reward count is known on the device only
  return EDP_OK;
}

edp_status edp_pack_deliver(edp_ctx *ctx, const int32_t *tokens, const uint64_t *seq_off,
                            uint64_t n_seq, const int64_t *idx, uint32_t batch,
                            const float *seq_value, int32_t *out_tokens,
                            uint64_t *out_off, float *out_value, uint64_t out_cap,
                            edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!tokens || !seq_off || !idx || !out_tokens || !out_off)
    return fail(ctx, EDP_ERR_INVALID, "edp_pack_deliver: NULL array");
  if (n_seq == 0 || batch == 0 || batch > (1u << 20))
    return fail(ctx, EDP_ERR_INVALID, "edp_pack_deliver: need n_seq > 0, 0 < batch <= 2^20");
  if ((seq_value == nullptr) != (out_value == nullptr))
    return fail(ctx, EDP_ERR_INVALID, "edp_pack_deliver: seq_value and out_value go together");
  const void *p;
  const void *ins[] = {tokens, seq_off, idx, seq_value};
  for (const void *o : ins)
    if (o && !device_view(ctx, o, &p, false))
      return fail(ctx, EDP_ERR_INVALID, "edp_pack_deliver: inputs must be device memory");
  void *outs[] = {out_tokens, out_off, out_value};
  for (void *&o : outs) {
    if (!o) continue;
    if (!device_view(ctx, o, &p, true))
      return fail(ctx, EDP_ERR_INVALID,
                  "edp_pack_deliver: outputs must be device or page-locked host memory");
    o = const_cast<void *>(p);
  }
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_pack(ctx, tokens, seq_off, n_seq, idx, batch, seq_value,
                              (int32_t *)outs[0], (uint64_t *)outs[1], (float *)outs[2],
                              out_cap, (cudaStream_t)stream);
  if (e != cudaSuccess) return launch_fail(ctx, e, "edp_pack_deliver");
  count_hbm(ctx, 24ull * batch, 0);  // indices and sequence offsets; tokens not counted
  count_write(ctx, out_off, 8ull * (batch + 1));
  ctx->cnt.delivered += batch;
  return EDP_OK;
}

edp_status edp_grpo_pack_deliver(edp_ctx *ctx, const float *r, const uint64_t *group_off,
                                 uint32_t n_groups, float eps, float *adv,
                                 const int32_t *tokens, const uint64_t *seq_off,
                                 uint64_t n_seq, const int64_t *idx, uint32_t batch,
                                 int32_t *out_tokens, uint64_t *out_off, float *out_value,
                                 uint64_t out_cap, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  if (!r || !group_off || !adv || n_groups == 0)
    return fail(ctx, EDP_ERR_INVALID, "edp_grpo_pack_deliver: NULL array or no group");
  if (!(eps >= 0.f) || !std::isfinite(eps))
    return fail(ctx, EDP_ERR_INVALID, "edp_grpo_pack_deliver: eps must be finite and >= 0");
  if (!tokens || !seq_off || !idx || !out_tokens || !out_off)
    return fail(ctx, EDP_ERR_INVALID, "edp_grpo_pack_deliver: NULL array");
  if (n_seq == 0 || batch == 0 || batch > (1u << 20))
    return fail(ctx, EDP_ERR_INVALID,
                "edp_grpo_pack_deliver: need n_seq > 0, 0 < batch <= 2^20");
  const void *p;
  const void *ins[] = {r, group_off, adv, tokens, seq_off, idx};
  for (const void *o : ins)
    if (o && !device_view(ctx, o, &p, false))
      return fail(ctx, EDP_ERR_INVALID, "edp_grpo_pack_deliver: arrays must be device memory");
  void *outs[] = {out_tokens, out_off, out_value};
  for (void *&o : outs) {
    if (!o) continue;
    if (!device_view(ctx, o, &p, true))
      return fail(ctx, EDP_ERR_INVALID,
                  "edp_grpo_pack_deliver: outputs must be device or page-locked host memory");
    o = const_cast<void *>(p);
  }
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = launch_grpo_pack(ctx, r, group_off, n_groups, eps, adv, tokens, seq_off,
                                   n_seq, idx, batch, (int32_t *)outs[0], (uint64_t *)outs[1],
                                   (float *)outs[2], out_cap, (cudaStream_t)stream);
  if (e != cudaSuccess) return launch_fail(ctx, e, "edp_grpo_pack_deliver");
  count_hbm(ctx, 8ull * (n_groups + 1) + 24ull * batch, 0);
  count_write(ctx, out_off, 8ull * (batch + 1));
  ctx->cnt.delivered += batch;
  return EDP_OK;
}

edp_status edp_get_counters(edp_ctx *ctx, edp_counters *out) {
  if (!ctx || !out) return EDP_ERR_INVALID;
  *out = ctx->cnt;
  if (ctx->cap_c) {  // two-tier: the host-tier bytes the deliveries counted
    DeviceGuard dg(ctx->cfg.device);
    unsigned long long hb = 0;
    const cudaError_t e = cudaMemcpy(&hb, &ctx->ctrl->host_bytes, sizeof hb,
                                     cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_get_counters");
    uint64_t d = hb - ctx->host_bytes_base;
    if (d > out->hbm_read) d = out->hbm_read;
    out->hbm_read -= d;
    out->link_read += d;
  }
  return EDP_OK;
}

edp_status edp_reset_counters(edp_ctx *ctx) {
  if (!ctx) return EDP_ERR_INVALID;
  ctx->cnt = edp_counters{};
  if (ctx->cap_c) {
    DeviceGuard dg(ctx->cfg.device);
    unsigned long long hb = 0;
    const cudaError_t e = cudaMemcpy(&hb, &ctx->ctrl->host_bytes, sizeof hb,
                                     cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_reset_counters");
    ctx->host_bytes_base = hb;
  }
  return EDP_OK;
}

edp_status edp_sync(edp_ctx *ctx, edp_stream stream) {
  if (!ctx) return EDP_ERR_INVALID;
  DeviceGuard dg(ctx->cfg.device);
  EDP_TRACE(__func__);
  cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
  if (e == cudaSuccess) e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_sync");
  Ctrl h;
  e = cudaMemcpy(&h, ctx->ctrl, sizeof h, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(ctx, e, "edp_sync(read flags)");
  if (h.err == 0) return EDP_OK;
  const uint32_t zero[2] = {0, 0};
  cudaMemcpy(&ctx->ctrl->err, zero, 4, cudaMemcpyHostToDevice);
  cudaMemcpy(&ctx->ctrl->bad_index, zero, 8, cudaMemcpyHostToDevice);
  const unsigned long long bi = h.bad_index ? h.bad_index - 1 : 0;
  if (h.err & DEVERR_TIMEOUT)
    return fail(ctx, EDP_ERR_TIMEOUT, "device: a bounded wait expired (flags 0x%x)", h.err);
  if (h.err & DEVERR_EMPTY)
    return fail(ctx, EDP_ERR_EMPTY, "device: total priority was 0 (flags 0x%x)", h.err);
  if (h.err & DEVERR_TREE)
    return fail(ctx, EDP_ERR_STATE, "device: inconsistent priority tree (flags 0x%x)", h.err);
  if (h.err & DEVERR_OVERFLOW)
    return fail(ctx, EDP_ERR_INVALID,
                "device: a packed output or a sum of shard totals exceeds its capacity "
                "(%llu, flags 0x%x)", bi, h.err);
  return fail(ctx, EDP_ERR_INVALID,
              "device: index out of range (first offender %llu, flags 0x%x)", bi, h.err);
}

edp_status edp_probe_host_read(const void *host_src, uint64_t bytes,
                               uint64_t *d_fold, edp_stream stream) {
  if (!host_src || !d_fold || bytes % 16) return EDP_ERR_INVALID;
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, host_src) != cudaSuccess) {
    cudaGetLastError();
    return EDP_ERR_INVALID;
  }
  const void *src = host_src;
  if (a.type == cudaMemoryTypeHost) src = a.devicePointer;
  else if (a.type != cudaMemoryTypeDevice) return EDP_ERR_INVALID;
  if (!src || !aligned16(src)) return EDP_ERR_INVALID;
  return launch_probe_read(src, bytes, d_fold, (cudaStream_t)stream) == cudaSuccess
             ? EDP_OK
             : EDP_ERR_CUDA;
}

}  // extern "C"
