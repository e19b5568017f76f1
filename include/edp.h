/*
 * edp.h -- C ABI of libedp, the GB300 (sm_103a) hot path of an Experience
 * Data Plane for distributed reinforcement learning.
 *
 * The paper (Conduit) exposes the experience path through three control
 * points -- ingestion, placement, delivery (Sec. 3, "Overview"; Sec. 2.2,
 * "Experience Path Responsibilities") -- plus the replay-state priority
 * callback (Appendix C, Invariant 2).  This header maps them to calls:
 *
 *   ingestion  -> edp_ingest            (ring scatter; two-tier demotion)
 *                 edp_gae               (on-policy returns/advantages)
 *   placement  -> edp_config.hbm_capacity / edp_storage.host_*  (two tiers)
 *   delivery   -> edp_sample            (uniform, prioritized, shuffle)
 *                 edp_deliver           (gather + transform + collate)
 *   callback   -> edp_update_priorities / edp_update_priorities_td
 *   sharding   -> edp_tree_total, edp_route_prioritized, edp_sample_targets,
 *                 edp_batch_qmin, edp_is_weights, edp_gae_stats,
 *                 edp_gae_normalize (a buffer split across GPUs, Sec. 5.1)
 *
 * Conventions shared by every call
 * --------------------------------
 * - Plain C types only.  A `edp_stream` is a cudaStream_t (NULL = the legacy
 *   default stream).  Pointers documented "device" must be device memory of
 *   the context's GPU; "device-accessible" also admits page-locked host
 *   memory (cudaHostAlloc / cudaHostRegister, e.g. torch pin_memory), which
 *   kernels then read or write over the host link.
 * - Ownership: the caller allocates and frees every buffer it passes (ring
 *   storage, inputs, outputs).  libedp owns only the context, the priority
 *   tree and small scratch, allocated through edp_config.alloc (cudaMalloc
 *   when NULL) and released by edp_destroy.  libedp never frees caller memory.
 *   Scratch is allocated at a call's first use and grown (after a device
 *   synchronisation) when a later call needs more: edp_update_priorities_td
 *   (4 bytes per pair), the PERMUTE sampling mode, edp_gae with
 *   normalisation and edp_pack_deliver (16 bytes per batch entry).  Before
 *   capturing calls into a CUDA graph, make each of them once at its
 *   largest size, outside the capture: a call that would have to grow its
 *   scratch while its stream is being captured returns EDP_ERR_STATE and
 *   enqueues nothing.
 * - Current device: a call makes its context's device current while it
 *   runs and gives the calling thread its previous current device back
 *   before it returns.
 * - Asynchrony: every call validates its arguments on the host, enqueues its
 *   kernels on `stream` and returns without synchronising.  Results are
 *   valid once the stream has reached that point.  Host-side cursors
 *   (head, total) advance at enqueue time, so calls on one context must be
 *   issued in program order on one stream (or with the caller's own
 *   cross-stream ordering).
 * - Overlap (the overlapped timing of Sec. 6.1): edp_deliver reads only the
 *   ring storage, its `idx` / `q` and the gather sources, and writes only
 *   its batch, so it may run on another stream concurrently with
 *   edp_sample, edp_update_priorities*, edp_priorities_from_td, edp_gae and
 *   other deliveries of the same context, once the sampling that wrote its
 *   `idx` has completed (an event) and while nothing overwrites `idx`, `q`
 *   or the rows it reads (edp_ingest).  Any number of deliveries may be in
 *   flight at once, on any streams or in one graph.
 *   edp_gae likewise may overlap edp_sample (GAE scratch and shuffle
 *   scratch are separate); edp_gae and edp_pack_deliver share scratch.
 *   Every other pair of calls on one context shares the priority tree or
 *   the context's scratch and must be ordered.
 * - Errors: argument and state errors are returned synchronously and leave
 *   the context unchanged.  A CUDA launch error returns EDP_ERR_CUDA.
 *   Data-dependent faults found on the device (an index out of range, an
 *   all-zero priority distribution, a bounded wait that expired) never trap:
 *   the kernel records a flag, writes zeros / -1 for the affected outputs and
 *   returns; edp_sync reports the flag.  No C++ exception crosses the ABI.
 *   edp_last_error() describes the last failure of a context.
 * - Randomness is stateless: each sampling call derives its draws from
 *   (seed, round, stream id) through Philox4x32-10 (Salmon et al., SC'11),
 *   so the same arguments give the same indices.
 */
#ifndef EDP_H
#define EDP_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define EDP_ABI_VERSION 2

/* Symbols of the ABI are exported; everything else in libedp is hidden. */
#if defined(__GNUC__)
#define EDP_API __attribute__((visibility("default")))
#else
#define EDP_API
#endif

typedef struct edp_ctx edp_ctx;  /* opaque; created by edp_create */
typedef void *edp_stream;        /* cudaStream_t */

typedef enum {
  EDP_OK = 0,
  EDP_ERR_INVALID = 1, /* bad argument, or a device-detected bad index */
  EDP_ERR_OOM = 2,     /* the allocator returned NULL */
  EDP_ERR_CUDA = 3,    /* a CUDA runtime error (launch or asynchronous) */
  EDP_ERR_TIMEOUT = 4, /* a bounded device-side wait expired */
  EDP_ERR_EMPTY = 5,   /* nothing to sample (no valid transition, or total
                          priority 0) */
  EDP_ERR_STATE = 6    /* call not valid for this context's configuration */
} edp_status;

/* How edp_deliver turns a stored uint8 observation into the learner layout.
 * All three divide by 255 as one correctly rounded binary32 division
 * x = fl32(b / 255); bfloat16 outputs are then rounded to nearest even. */
typedef enum {
  /* DQN-style frame stack (frame stacking of Mnih et al., Nature 2015):
   * obs[b][m] = frame of logical offset i-K+1+m, next_obs[b][m] = that of
   * i-K+2+m; a frame is all zeros when it precedes the oldest stored
   * transition or an episode end (done == 1) lies between it and the anchor
   * (exclusive of the anchor).  Output float32 [B][K][obs_h][obs_w]. */
  EDP_XFORM_STACK_F32 = 0,
  /* Stored HWC (obs_h x obs_w x obs_c), delivered CHW bfloat16
   * [B][obs_c][obs_h][obs_w] = RNE_bf16(x). */
  EDP_XFORM_HWC_CHW_BF16 = 1,
  /* Stored CHW, delivered bfloat16 [B][obs_c][obs_h][obs_w] =
   * RNE_bf16(fl32(fl32(x - mean_c) / std_c)), each step rounded. */
  EDP_XFORM_CHW_NORM_BF16 = 2
} edp_transform;

typedef enum {
  /* index_k = slot of logical offset mulhi64(u64(k; seed, round, 0), n_valid)
   * where n_valid = size - 1 when next_obs is delivered, else size. */
  EDP_SAMPLE_UNIFORM = 0,
  /* PER proportional sampling, stratified (Schaul et al., ICLR'16): with
   * S = total priority, stratum k of B targets t_k = lo_k + mulhi64(u64(k;
   * seed, round, 1), hi_k - lo_k), lo_k = floor(k S / B), hi_k =
   * floor((k+1) S / B); the answer is the slot whose priority interval
   * [prefix(i), prefix(i) + q_i) over physical slot order holds t_k. */
  EDP_SAMPLE_PRIORITIZED = 1,
  /* Shuffle of all `size` stored transitions (on-policy mini-batching):
   * logical offsets sorted by (u64(j; seed, round, 2), j); idx[r] = slot of
   * the r-th.  Mini-batch m of size M is idx[mM, (m+1)M). */
  EDP_SAMPLE_PERMUTE = 2
} edp_sample_mode;

/* Allocator for libedp-owned device memory (256-byte aligned).  Returning
 * NULL makes the calling function fail with EDP_ERR_OOM. */
typedef void *(*edp_alloc_fn)(void *user, size_t bytes);
typedef void (*edp_free_fn)(void *user, void *ptr);

typedef struct {
  uint64_t capacity;     /* logical ring capacity in transitions, 1..2^32-1 */
  uint64_t hbm_capacity; /* transitions whose payload (obs, tokens) lives in
                            HBM.  == capacity: single tier.  < capacity:
                            two-tier ring -- the newest hbm_capacity
                            transitions in HBM, the older ones in page-locked
                            host memory; requires transform CHW_NORM_BF16 */
  uint32_t obs_c, obs_h, obs_w; /* stored observation shape; obs_bytes =
                            c*h*w must be a multiple of 16 */
  uint32_t transform;    /* edp_transform */
  uint32_t frame_stack;  /* K for STACK_F32 (1..16); must be 1 otherwise */
  uint32_t next_obs;     /* STACK_F32 only: 1 = deliver next_obs as well; the
                            newest transition is then not sampleable */
  uint32_t tokens;       /* int32 tokens stored per transition (0 = none);
                            a multiple of 4 */
  uint32_t prioritized;  /* 1 = keep the priority sum-tree (PER) */
  float norm_mean[4];    /* CHW_NORM_BF16 per-channel mean (of byte/255) */
  float norm_std[4];     /* CHW_NORM_BF16 per-channel std, > 0 */
  edp_alloc_fn alloc;    /* NULL = cudaMalloc */
  edp_free_fn free;      /* NULL = cudaFree */
  void *alloc_user;
  int32_t device;        /* CUDA device ordinal of every device pointer */
  uint32_t reserved[7];  /* must be 0 */
} edp_config;

/* Caller-owned ring storage.  Slot s of the logical ring holds the
 * transition with logical id L where L mod capacity == s.  Its payload lives
 * in HBM slot L mod hbm_capacity or, for the two-tier ring, in host slot
 * L mod (capacity - hbm_capacity); metadata is HBM-resident for every slot. */
typedef struct {
  uint8_t *obs;         /* device [hbm_capacity][obs_bytes], 16-B aligned */
  int32_t *tokens;      /* device [hbm_capacity][tokens]; NULL iff tokens==0 */
  uint8_t *host_obs;    /* page-locked host [capacity-hbm_capacity][obs_bytes]
                           (two-tier only, else NULL), 16-B aligned */
  int32_t *host_tokens; /* page-locked host [capacity-hbm_capacity][tokens] */
  int32_t *action;      /* device [capacity] or NULL */
  float *reward;        /* device [capacity] or NULL */
  uint8_t *done;        /* device [capacity]; required for STACK_F32 */
} edp_storage;

/* n transitions to insert, logical order.  Device-accessible pointers. */
typedef struct {
  const uint8_t *obs;    /* [n][obs_bytes], 16-B aligned; required */
  const int32_t *tokens; /* [n][tokens]; required iff tokens > 0 */
  const int32_t *action; /* [n] or NULL (stores 0) */
  const float *reward;   /* [n] or NULL (stores 0) */
  const uint8_t *done;   /* [n] or NULL (stores 0) */
} edp_fields;

/* Learner batch written by edp_deliver.  NULL skips an output.  Outputs
 * (obs, next_obs, action, reward, done, tokens, isw, gather_dst) are device
 * memory, or page-locked host memory that the kernel then writes over the
 * host link (a learner on the host gets its batch with no separate copy);
 * the inputs q and gather_src are device memory.  B = the `batch` argument
 * of edp_deliver. */
typedef struct {
  void *obs;      /* see edp_transform; required */
  void *next_obs; /* STACK_F32 with next_obs == 1: float [B][K][h][w] */
  int32_t *action;
  float *reward;
  uint8_t *done;  /* [B] each, of the sampled (anchor) transition */
  int32_t *tokens;/* [B][tokens] */
  /* Importance-sampling weights (PER): isw[b] = (q_min / q[b])^beta with
   * q_min the minimum of q over the batch; fp64, rounded once to fp32.
   * q = the priorities edp_sample(PRIORITIZED) returned for this batch. */
  const uint32_t *q;
  float *isw;
  double beta;
  /* Per-sample scalars gathered by the sample's logical offset k (0 = the
   * oldest stored transition): dst[b] = src[k].  Used for the advantages and
   * returns of an on-policy rollout.  NULL pairs are skipped. */
  const float *gather_src[2];
  float *gather_dst[2];
} edp_batch;

/* Inspection of a context (host values, device pointers). */
typedef struct {
  uint64_t capacity, hbm_capacity, total, size, head, oldest, n_valid;
  uint32_t tree_depth;          /* D: leaves are level D, the root level 0 */
  uint32_t tree_fanout;         /* 32 */
  const uint32_t *tree_leaves;  /* device [32^D] */
  const uint64_t *tree_level[8];/* device; level d has 32^d nodes, d < D */
  const uint32_t *pending_q;    /* device [1]: deferred priority of newest */
  const uint32_t *max_q;        /* device [1]: running maximum priority */
  /* CHW_NORM_BF16: how the kernel evaluates the per-byte normalisation,
   * each form checked at creation against the exact chain for all 256 bytes
   * of every channel: 2 = one FMA, bf16(fma(b, A_c, B_c)) with A_c, B_c
   * within a few ulps of 1/(255 std_c) and -mean_c/std_c; 1 = the chain
   * with the division as an FMA by a split reciprocal; 0 = the chain with
   * IEEE division (also for other transforms). */
  uint32_t norm_path;
} edp_info;

/* Create a context on cfg->device over caller storage.  Fails with
 * EDP_ERR_INVALID for inconsistent shapes or pointers, EDP_ERR_OOM when the
 * allocator fails.  Synchronous (initialises the tree). */
EDP_API edp_status edp_create(const edp_config *cfg, const edp_storage *st,
                      edp_ctx **out);

/* Free libedp-owned memory.  Waits for the device to finish with it.
 * EDP_ERR_INVALID for a NULL context. */
EDP_API edp_status edp_destroy(edp_ctx *ctx);

/* Ingestion (Sec. 2.2 "experience ingestion", off-policy insertion with
 * FIFO eviction; Sec. 5 placement).  Inserts n (0..capacity) transitions at
 * logical ids total .. total+n-1.  Two-tier ring: first moves the payload of
 * the oldest HBM-resident transitions that must leave HBM into the host tier
 * (evicting the oldest host entries), then writes the new payload to HBM.
 * PER: q (device [n] or NULL) gives each new transition's priority (NULL =
 * the running maximum, initially 2^20 = 1.0).  With next_obs, the newest
 * transition's priority is deferred until its successor arrives.
 * Errors: EDP_ERR_INVALID when n > capacity, src or src->obs is NULL, a
 * field is neither device nor page-locked memory, obs or tokens are not
 * 16-byte aligned, tokens are given to a context without tokens (or
 * missing for one with them), or q is not device memory; EDP_ERR_STATE for
 * q on a context without priorities; EDP_ERR_CUDA when a launch fails.
 * n == 0 does nothing. */
EDP_API edp_status edp_ingest(edp_ctx *ctx, const edp_fields *src, uint64_t n,
                      const uint32_t *q, edp_stream stream);

/* Sampling (Sec. 2.2: choosing which stored transitions a batch holds).
 * Writes idx (device int64 [batch])
 * and, for PRIORITIZED, q (device uint32 [batch], may be NULL) = the sampled
 * leaves.  Errors: EDP_ERR_EMPTY when no transition is sampleable;
 * EDP_ERR_STATE for PRIORITIZED without a tree; EDP_ERR_INVALID when
 * batch == 0 or, for PERMUTE, batch != size. */
EDP_API edp_status edp_sample(edp_ctx *ctx, edp_sample_mode mode, uint32_t batch,
                      uint64_t seed, uint64_t round, int64_t *idx,
                      uint32_t *q, edp_stream stream);

/* Delivery (Sec. 2.2: the chosen transitions are materialised in the
 * learner's batch layout): fused gather + transform + collate (+ IS
 * weights) of the `batch` slots in idx (device int64).  A slot outside the
 * sampleable range is reported by edp_sync and its outputs are zeroed.
 * The batch's outputs may be device or page-locked host memory (edp_batch).
 * Errors: EDP_ERR_INVALID for a NULL idx, out or out->obs, batch == 0,
 * inputs (idx, q, gather sources) outside device memory, outputs neither
 * device nor page-locked memory, obs / next_obs / tokens not 16-byte
 * aligned, isw without q or with beta < 0, or a half-NULL gather pair;
 * EDP_ERR_EMPTY for an empty ring; EDP_ERR_STATE for an output the context
 * does not store (next_obs without next_obs = 1, tokens, action, reward,
 * done). */
EDP_API edp_status edp_deliver(edp_ctx *ctx, const int64_t *idx, uint32_t batch,
                       const edp_batch *out, edp_stream stream);

/* Fused uniform sample -> deliver: the UNIFORM draw of edp_sample (same seed,
 * round, indices) made inside the delivery kernel, one launch instead of
 * two.  idx (device int64 [batch]) receives the drawn slots; out as for
 * edp_deliver, without q / isw (uniform draws carry no priorities:
 * EDP_ERR_INVALID).  EDP_ERR_EMPTY when no transition is sampleable; other
 * errors as edp_deliver.  Prioritized sampling keeps its own kernel, whose
 * tree descents every delivery warp would otherwise repeat. */
EDP_API edp_status edp_sample_deliver(edp_ctx *ctx, uint32_t batch, uint64_t seed,
                                      uint64_t round, int64_t *idx, const edp_batch *out,
                                      edp_stream stream);

/* Priority callback (Appendix C, Invariant 2; PER).  Sets the priority of
 * each (idx[p], q[p]); for a repeated slot the last pair wins.  Pairs whose
 * slot holds no transition are skipped; the newest transition's priority is
 * deferred (next_obs).  Ancestor sums change by exact integer deltas.
 * Errors: EDP_ERR_STATE for a context without priorities; EDP_ERR_INVALID
 * for NULL inputs or inputs outside device memory (and, for the TD forms,
 * alpha or eps < 0); EDP_ERR_OOM when the TD form cannot allocate its
 * scratch.  n == 0 does nothing. */
EDP_API edp_status edp_update_priorities(edp_ctx *ctx, const int64_t *idx,
                                 const uint32_t *q, uint32_t n,
                                 edp_stream stream);

/* Same, from TD errors: q = clamp(rn((|td| + eps)^alpha * 2^20), 1,
 * 2^32-1), the rule defined in fp64.  For alpha in (0, 1] and |td| + eps in
 * [2^-100, 2^100] the device evaluates it in double-float arithmetic
 * (relative error below 2^-40), otherwise in fp64; neither is correctly
 * rounded, so q may differ by 1 from a host evaluation (about one case in
 * a million).  Batches of up to 2048 pairs need no scratch. */
EDP_API edp_status edp_update_priorities_td(edp_ctx *ctx, const int64_t *idx,
                                    const float *td, uint32_t n, double alpha,
                                    double eps, edp_stream stream);

/* edp_update_priorities_td without any device allocation.  The paper has no
 * counterpart: this entry point exists for callers that cannot allocate
 * device memory when they update priorities -- code being captured into a
 * CUDA graph, where cudaMalloc may not be called, and runtimes that hand out
 * all device memory at start-up and forbid later allocation, or cannot
 * afford the device-wide synchronisation an allocation may bring.
 * Above 2048 pairs edp_update_priorities_td allocates its scratch (one
 * uint32 per pair) on first use; this variant keeps that scratch in a fixed
 * per-device array of 16384 pairs (64 KiB), held by every GPU that loads
 * libedp until the process exits.  n > 16384 returns EDP_ERR_INVALID.  The first call on a device
 * looks up the array's device address (make it before any stream capture).
 * All calls on a device share the array.  Calls queued on one stream are
 * ordered (a call touches the array only after the previous kernel on its
 * stream has finished), so they may follow each other with no
 * synchronisation; calls that can run at the same time on different streams
 * -- of one context or of several on the device -- race on the array and
 * must be ordered by the caller (an event).  The array keeps the last call's
 * contents, which a call never reads before writing.  Results equal those of
 * edp_update_priorities_td for the same arguments. */
EDP_API edp_status edp_update_priorities_td_static(edp_ctx *ctx, const int64_t *idx,
                                                   const float *td, uint32_t n,
                                                   double alpha, double eps,
                                                   edp_stream stream);

/* The TD-error rule alone: q[i] from td[i] (device arrays [n]). */
EDP_API edp_status edp_priorities_from_td(edp_ctx *ctx, const float *td, uint32_t n,
                                  double alpha, double eps, uint32_t *q,
                                  edp_stream stream);

/* Generalized advantage estimation (Schulman et al., ICLR'16) -- the return
 * and advantage computation and their normalisation, steps of on-policy
 * ingestion (Sec. 2.2).  Device arrays, time-major: r, d [T][E]; v [T+1][E].
 *   delta_t = r_t + gamma V_{t+1} (1 - d_t) - V_t
 *   A_t = delta_t + gamma lambda (1 - d_t) A_{t+1},  A_T = 0
 *   ret_t = A_t + V_t
 *   adv_norm = (A - mean(A)) / (std(A) + 1e-8), std with n-1, over T*E
 * Computed in fp64, stored fp32 [T][E].  adv/ret/adv_norm may be NULL
 * individually.  T, E >= 1 and T*E < 2^31 (else EDP_ERR_INVALID); with a
 * single value (T*E == 1) the spread is 0 and adv_norm is 0. */
EDP_API edp_status edp_gae(edp_ctx *ctx, const float *r, const float *v,
                   const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                   double lambda, float *adv, float *ret, float *adv_norm,
                   edp_stream stream);

/* ---------------------------------------------------------------------------
 * Sharded buffer (Sec. 5.1, the shared-GPU placement: a node's GPUs each hold
 * a share of the ring's slots and every learner samples the whole buffer, so
 * most of a batch is fetched from other GPUs).  G ranks each hold one
 * context (a shard).  The global prioritized distribution is that of one
 * buffer whose leaves are the shards' leaves in shard-major order (all of
 * shard 0's physical slots, then shard 1's, ...), so a shard holds a
 * contiguous block of the global inverse CDF.  One round, for a global batch
 * of B split into consecutive strata per learner:
 *   1. edp_tree_total on every shard; the caller all-gathers the G totals;
 *   2. each learner: edp_route_prioritized over its strata -> local targets,
 *      grouped by owning shard, and per-shard counts; the caller exchanges
 *      the counts and then the targets (all-to-all);
 *   3. each owner: edp_sample_targets on the targets it received, in source
 *      rank order, then edp_deliver of those slots; the caller sends the rows
 *      (and slots and priorities) back with the reverse all-to-all -- they
 *      arrive at each learner in stratum order;
 *   4. each learner: edp_batch_qmin, a minimum over ranks by the caller, and
 *      edp_is_weights with that global minimum;
 *   5. priority updates travel to the owners in the same grouping and are
 *      applied with edp_update_priorities* (source rank order = global batch
 *      order, so the last occurrence of a slot still wins).
 * The indices, priorities, weights and rows equal those of a single buffer
 * holding all shards' leaves.  For on-policy rollouts sharded by
 * environment, edp_gae_stats gives each rank's (n, sum A, sum A^2); the
 * caller sums them over the ranks and edp_gae_normalize normalises with the
 * totals.  These calls never communicate: the exchanges are the caller's
 * (e.g. NCCL through torch.distributed).
 * ------------------------------------------------------------------------- */

/* Total priority S of this context's tree (device uint64 [1]).
 * EDP_ERR_STATE for a context without priorities; EDP_ERR_INVALID when
 * d_total is not device memory. */
EDP_API edp_status edp_tree_total(edp_ctx *ctx, uint64_t *d_total, edp_stream stream);

/* Stratified targets of strata k0 .. k0+n-1 of a global batch of `batch`
 * over G shard totals (device uint64 [G], shard order), as edp_sample
 * (PRIORITIZED) draws them over a single buffer (same seed, round and Philox
 * stream), each routed to the shard whose prefix range holds it:
 * d_local_t[i] (device uint64 [n]) = target - (totals of the shards before
 * the owner), in stratum order -- which groups them by owner, ascending --
 * and d_counts[s] (device int64 [G]) = strata owned by shard s.  The
 * context only names the GPU and receives device-side flags: an all-zero
 * total (DEVERR_EMPTY, edp_sync -> EDP_ERR_EMPTY) or a sum of totals beyond
 * 64 bits (DEVERR_OVERFLOW) routes nothing (counts 0, targets 2^64-1).
 * EDP_ERR_INVALID when G is 0 or above 1024, batch is 0, k0 + n > batch, or
 * a pointer is not device memory. */
EDP_API edp_status edp_route_prioritized(edp_ctx *ctx, const uint64_t *d_totals, uint32_t G,
                                         uint32_t batch, uint32_t k0, uint32_t n,
                                         uint64_t seed, uint64_t round, uint64_t *d_local_t,
                                         int64_t *d_counts, edp_stream stream);

/* Tree descent of n given targets (device uint64 [n], each below this
 * shard's total): d_idx (device int64 [n]) = the physical slot whose
 * prefix range holds the target, d_q (device uint32 [n] or NULL) = its
 * priority.  A target at or above the total gives idx -1, q 0 and a device
 * flag (edp_sync -> EDP_ERR_INVALID).  EDP_ERR_STATE without priorities;
 * EDP_ERR_INVALID for pointers outside device memory.  n == 0 does nothing. */
EDP_API edp_status edp_sample_targets(edp_ctx *ctx, const uint64_t *d_targets, uint32_t n,
                                      int64_t *d_idx, uint32_t *d_q, edp_stream stream);

/* Minimum of d_q[0..n) (device uint32) into d_qmin (device int64 [1]);
 * 2^32 - 1 for n == 0.  EDP_ERR_INVALID for pointers outside device memory. */
EDP_API edp_status edp_batch_qmin(edp_ctx *ctx, const uint32_t *d_q, uint32_t n,
                                  int64_t *d_qmin, edp_stream stream);

/* Importance weights of a batch whose priority minimum is given:
 * d_w[k] = (q_min / d_q[k])^beta in fp64, rounded once to fp32, with q_min =
 * *d_qmin (device int64, e.g. the minimum over every rank's share of a global
 * batch) -- the weights edp_deliver computes with q_min over its own batch.
 * EDP_ERR_INVALID for beta < 0 or pointers outside device memory.  n == 0
 * does nothing. */
EDP_API edp_status edp_is_weights(edp_ctx *ctx, const uint32_t *d_q, uint32_t n,
                                  const int64_t *d_qmin, double beta, float *d_w,
                                  edp_stream stream);

/* edp_gae without the normalisation, for environments sharded over ranks:
 * writes adv (required) and ret (or NULL) as edp_gae does, and d_stats
 * (device double [3]) = (T*E, sum of A, sum of A^2) over this rank's
 * values.  Errors as edp_gae, and EDP_ERR_INVALID when adv or d_stats is
 * NULL. */
EDP_API edp_status edp_gae_stats(edp_ctx *ctx, const float *r, const float *v,
                                 const uint8_t *d, uint32_t T, uint32_t E, double gamma,
                                 double lambda, float *adv, float *ret, double *d_stats,
                                 edp_stream stream);

/* adv_norm[i] = (adv[i] - mean) / (std + 1e-8) for i < n, with mean and the
 * unbiased std from d_stats = (N, sum A, sum A^2) (device double [3]: the
 * sums of every rank's edp_gae_stats); N == 1 gives 0.  adv and adv_norm
 * device float [n] (they may be the same array).  EDP_ERR_INVALID for n == 0,
 * n >= 2^31 or pointers outside device memory. */
EDP_API edp_status edp_gae_normalize(edp_ctx *ctx, const float *adv, uint64_t n,
                                     const double *d_stats, float *adv_norm,
                                     edp_stream stream);

/* ---------------------------------------------------------------------------
 * LLM post-training (Appendix A, Table "Verl map"): advantage computation is
 * part of ingestion; the hand-off of variable-length sequences is delivery
 * (Sec. 2.2 names padding / packing of variable-length sequences among the
 * delivery operators).  Any context of the GPU serves for error reporting;
 * its ring is not used.
 * ------------------------------------------------------------------------- */

/* Group-relative advantages (GRPO, Shao et al. 2024): responses to one prompt
 * form a group, g = [group_off[g], group_off[g+1]); for i in g
 *   A_i = (r_i - mean_g) / (std_g + eps),
 * std_g the sample standard deviation (divisor n_g - 1; 0 for n_g = 1).
 * Computed in fp64, stored fp32; A_i = 0 where std_g + eps = 0.  r, adv:
 * device float[group_off[n_groups]]; group_off: device uint64[n_groups + 1],
 * non-decreasing, group_off[0] = 0.  A group of equal rewards gets A = 0.
 * Errors: EDP_ERR_INVALID for a NULL array, n_groups == 0, eps negative or
 * not finite, or arrays outside device memory. */
EDP_API edp_status edp_grpo_advantage(edp_ctx *ctx, const float *r,
                                      const uint64_t *group_off, uint32_t n_groups,
                                      float eps, float *adv, edp_stream stream);

/* Packed delivery of variable-length sequences (the "varlen" layout):
 * sequence s of tokens (device int32) is [seq_off[s], seq_off[s+1]),
 * seq_off device uint64[n_seq + 1] non-decreasing.  For the batch
 * idx[0..batch) (device int64, any order, repeats allowed):
 *   out_off[k]  = sum_{j<k} len(idx[j])              (uint64[batch + 1])
 *   out_tokens[out_off[k] + t] = tokens[seq_off[idx[k]] + t]
 *   out_value[out_off[k] + t]  = seq_value[idx[k]]   (optional: a per-
 *                       sequence value, e.g. its advantage, on every token)
 * out_cap: elements available in out_tokens / out_value.  An index outside
 * [0, n_seq) delivers an empty sequence; output beyond out_cap is not
 * written; both set a device flag that edp_sync reports (EDP_ERR_INVALID;
 * for an overflow the message gives the size needed).  batch <= 2^20.
 * The outputs (out_tokens, out_off, out_value) may be page-locked host
 * memory, written over the host link; the inputs are device memory.
 * Errors: EDP_ERR_INVALID for a NULL array, n_seq == 0, batch == 0 or
 * > 2^20, seq_value without out_value (or the reverse), inputs outside
 * device memory, or outputs neither device nor page-locked memory;
 * EDP_ERR_OOM when the batch's scratch cannot be allocated. */
EDP_API edp_status edp_pack_deliver(edp_ctx *ctx, const int32_t *tokens,
                                    const uint64_t *seq_off, uint64_t n_seq,
                                    const int64_t *idx, uint32_t batch,
                                    const float *seq_value, int32_t *out_tokens,
                                    uint64_t *out_off, float *out_value, uint64_t out_cap,
                                    edp_stream stream);

/* The GRPO step in one call: the group-relative advantages of
 * edp_grpo_advantage (r, group_off, n_groups, eps -> adv) and the packed
 * delivery of edp_pack_deliver with seq_value = adv, so sequence s is
 * response s (n_seq = group_off[n_groups]; adv has n_seq entries).  The
 * advantages are computed beside the batch's length pass (the two are
 * independent until the copy), then the copy puts each response's advantage
 * on its tokens; out_value may be NULL (advantages only written to adv).
 * Same results, scratch use and errors as the two calls. */
EDP_API edp_status edp_grpo_pack_deliver(edp_ctx *ctx, const float *r,
                                         const uint64_t *group_off, uint32_t n_groups,
                                         float eps, float *adv, const int32_t *tokens,
                                         const uint64_t *seq_off, uint64_t n_seq,
                                         const int64_t *idx, uint32_t batch,
                                         int32_t *out_tokens, uint64_t *out_off,
                                         float *out_value, uint64_t out_cap,
                                         edp_stream stream);

/* Wait for `stream`, then report (and clear) asynchronous CUDA errors and
 * device-side flags recorded since the previous edp_sync. */
EDP_API edp_status edp_sync(edp_ctx *ctx, edp_stream stream);

/* Describe the context's last failure ("" if none).  Valid until the next
 * call on the context.  "null context" for NULL. */
EDP_API const char *edp_last_error(const edp_ctx *ctx);

/* Online placement migration (Sec. 5.3, Alg. 2): move the experience state
 * of `src` into `dst`, a context created empty with the new placement --
 * another hbm_capacity (GPU only <-> GPU + host tier) or another capacity
 * -- and the same transform, observation shape, frame_stack, next_obs,
 * tokens, prioritized flag, metadata arrays and device.  dst receives the
 * newest n = min(size, dst capacity) transitions, oldest first, as if they
 * had been its first n insertions (its total becomes n, so slots change:
 * indices sampled from src do not apply to dst): payload rows go from
 * their tier in src to their tier in dst (HBM or page-locked host, every
 * direction in one launch, Appendix D), action / reward / done and
 * priority leaves along, and the deferred and maximum priorities; dst's
 * tree is rebuilt.  src is left unchanged.  The two must not share storage, and
 * nothing may write src or use dst on another stream until `stream` has
 * passed this call.  EDP_ERR_STATE when dst is not empty or the layouts
 * differ. */
EDP_API edp_status edp_migrate(const edp_ctx *src, edp_ctx *dst, edp_stream stream);

/* Checkpoint / resume (no counterpart in the paper, which keeps no
 * fault tolerance; an experience buffer worth hours of rollouts is worth
 * saving).  edp_save waits for `stream`, then writes the context's
 * retained transitions in logical order -- payload rows from both tiers,
 * action / reward / done, priority leaves, the deferred and maximum
 * priorities -- with a header describing the layout, to the file `path`.
 * edp_load reads such a file into an empty context of the same layout
 * (transform, observation shape, frame_stack, next_obs, tokens,
 * prioritized flag, metadata arrays); capacity and tier split may differ:
 * the newest min(saved, capacity) transitions become its first insertions,
 * placed by its own tier map, and its tree is rebuilt on `stream`.  Both
 * stage the data through 64 MiB of host memory and synchronise.
 * EDP_ERR_INVALID for an unreadable or foreign file, or one whose size is
 * not the size its header describes (checked before anything is written;
 * after a later read error the context is reset to empty, priorities
 * included), EDP_ERR_STATE for a non-empty context or another layout. */
EDP_API edp_status edp_save(edp_ctx *ctx, const char *path, edp_stream stream);
EDP_API edp_status edp_load(edp_ctx *ctx, const char *path, edp_stream stream);

/* Fill *out with the context's cursors and tree layout.  EDP_ERR_INVALID
 * for a NULL argument. */
EDP_API edp_status edp_get_info(const edp_ctx *ctx, edp_info *out);

/* Per-context traffic counters (no counterpart in the paper, whose metrics
 * are latencies).  Counts accumulate from context creation or the last
 * edp_reset_counters, at enqueue time, for every call that enqueued work.
 * Byte counts are algorithmic, the bytes the path must move: the payload
 * rows and metadata an insertion reads from its source and writes to the
 * ring (demotions included), the source bytes a delivery reads and the
 * outputs it writes, and the index / priority arrays of sampling and
 * updates.  Every count is split by where the bytes live: device memory
 * (hbm_*) or page-locked host memory reached over the host link (link_*).
 * The tier of a two-tier delivery's rows depends on the sampled slots, so
 * its kernel counts its host-tier rows on the device; edp_get_counters
 * reads that count, which is exact once the deliveries have completed
 * (e.g. after edp_sync).  Not counted: a packed delivery's tokens, whose
 * number is only known on the device, and traffic inside the priority tree.
 * EDP_ERR_INVALID for a NULL argument; EDP_ERR_CUDA when the device count
 * cannot be read. */
typedef struct {
  uint64_t calls;       /* calls that enqueued work */
  uint64_t ingested;    /* transitions inserted */
  uint64_t sampled;     /* indices drawn (sampling, fused sampling) */
  uint64_t delivered;   /* batch entries delivered */
  uint64_t hbm_read, hbm_write;    /* bytes read from / written to device memory */
  uint64_t link_read, link_write;  /* bytes read from / written to host memory */
} edp_counters;
EDP_API edp_status edp_get_counters(edp_ctx *ctx, edp_counters *out);
EDP_API edp_status edp_reset_counters(edp_ctx *ctx);

/* Host-link probe: streams `bytes` (a multiple of 16) of page-locked host
 * memory through the GPU with 16-byte loads, xor-folding them into
 * *d_fold (device uint64).  Used to measure achievable host-link read
 * bandwidth for the two-tier ring.  Takes no context.  EDP_ERR_INVALID for
 * NULL pointers, bytes not a multiple of 16, or a source that is not
 * 16-byte aligned page-locked host or device memory; EDP_ERR_CUDA when the
 * launch fails. */
EDP_API edp_status edp_probe_host_read(const void *host_src, uint64_t bytes,
                               uint64_t *d_fold, edp_stream stream);

/* ---------------------------------------------------------------------------
 * Latency-aware scheduling (Sec. 6): choose when ingestion and delivery run
 * (timing: inline, or overlapped with rollout / learner update) and how much
 * each invocation processes (granularity g: g >= 1 batches g rollout units /
 * training batches, 0 < g < 1 pipelines a fraction of one), from profiled
 * costs, by the iteration-latency model of Sec. 6.2 and Appendix E and the
 * enumeration of Eq. 2 (Sec. 6.3):
 *
 *   Tbar(g)    = T(g) / g                       (per-unit cost)
 *   gamma(g)   = 1 if g >= 1, else 1 - g
 *   hide_ing   = (1 - c_ing) gamma(g_ing) min(T_rollout, Tbar_ing(g_ing))
 *   hide_del   = (1 - c_del) gamma(g_del) min(T_update,  Tbar_del(g_del))
 *   T_ing_path = T_rollout + Tbar_ing(g_ing) + o_ing (T_sync_ing - hide_ing)
 *   T_del_path = T_update  + Tbar_del(g_del) + o_del (T_sync_del - hide_del)
 *   T_iter     = T_ing_path + T_del_path,  minimised over o_ing, o_del in
 *                {0, 1} and the candidate granularities.
 *
 * c_ing, c_del are not in the paper, which assumes the hidden part of an
 * operator costs its neighbour nothing; they are 0 there (the default of a
 * zeroed struct).  On one GPU the delivery and the learner update contend
 * for the same SMs and HBM, so only part of the overlap hides: a caller
 * that measured it passes the contention c in [0, 1].
 *
 * Host-only: no GPU work, no context.  Times in any one unit.
 * ------------------------------------------------------------------------- */
typedef struct {
  double t_rollout;      /* one actor rollout */
  double t_update;       /* one learner update */
  double t_sync_ing;     /* synchronisation added by overlapping ingestion */
  double t_sync_del;     /* ... by overlapping delivery */
  uint32_t n_ing, n_del; /* number of candidate granularities (>= 1 each) */
  const double *g_ing;   /* [n_ing] candidate g_ing, each > 0 */
  const double *t_ing;   /* [n_ing] T_ing(g): one invocation's wall time */
  const double *g_del;   /* [n_del] candidate g_del, each > 0 */
  const double *t_del;   /* [n_del] T_del(g) */
  double contention_ing; /* c_ing in [0, 1]: share of the hidden time lost */
  double contention_del; /* c_del in [0, 1] */
} edp_sched_costs;

typedef struct {
  uint32_t overlap_ing, overlap_del; /* timing flags, 0 or 1 */
  uint32_t i_ing, i_del;             /* indices of the chosen granularities */
  double g_ing, g_del;
  double t_ing_path, t_del_path, t_iter;
} edp_sched_choice;

/* Score every candidate (o_ing, o_del, i_ing, i_del) and write the one with
 * the lowest T_iter to *best; ties keep the first in the order o_ing,
 * o_del, i_ing, i_del, each ascending (so inline timing and the earlier
 * candidate win a tie).  t_iter_all (may be NULL) receives every score,
 * [2][2][n_ing][n_del] in that order.  EDP_ERR_INVALID for a NULL argument,
 * a zero count, a non-positive or non-finite g, a negative or non-finite
 * time, or a contention outside [0, 1]. */
EDP_API edp_status edp_sched_choose(const edp_sched_costs *costs,
                                    edp_sched_choice *best, double *t_iter_all);

/* Candidate granularities derived from the RL configuration (Sec. 6.3):
 * off-policy (on_policy = 0): 1, 2, 4, ... up to `m` batches per invocation;
 * on-policy: k / m for every divisor k of m, m = mini-batches per rollout
 * unit, ascending.  Writes at most `cap` values to g and returns how many
 * there are (call with cap = 0 to size g); 0 if m == 0. */
EDP_API uint32_t edp_sched_granularities(uint32_t on_policy, uint32_t m, double *g,
                                         uint32_t cap);

/* ---------------------------------------------------------------------------
 * Bandwidth-aware placement (Sec. 5): the per-sample transfer latency of a
 * placement p (Sec. 5.1)
 *
 *   T(p, x) = x / BW(actor -> p) + x / BW(p -> learner GPU)
 *
 * and the feasible minimum of Eq. 1, found by the linear scan of Alg. 1:
 * p* = argmin T(p, x) subject to C_buf x <= Mem(p); the first option wins a
 * tie.  A placement may have two tiers (the paper's mixture of local and
 * remote reads, here fast and slow memory of one node): the newest
 * transitions fill tier 1, so with uniform sampling a share
 * h = min(1, Mem1 / (C_buf x)) of the reads comes from tier 1 and
 *
 *   x / BW(p -> GPU) = x (h / bw_out + (1 - h) / bw_out2),
 *
 * feasible when C_buf x <= Mem1 + Mem2.  Bandwidths in bytes/s, sizes in
 * bytes, times in seconds.  Host-only: no GPU work, no context.
 * ------------------------------------------------------------------------- */
typedef enum {
  EDP_PLACE_HOST_PAGEABLE = 0, /* CPU pageable memory (staged copies) */
  EDP_PLACE_HOST_PINNED = 1,   /* CPU page-locked memory, zero-copy reads */
  EDP_PLACE_GPU = 2,           /* HBM of the learner's GPU */
  EDP_PLACE_GPU_HOST = 3       /* newest in HBM, older in page-locked memory */
} edp_place_kind;

typedef struct {
  uint32_t kind;      /* edp_place_kind; not used by the arithmetic */
  uint32_t tiers;     /* 1 or 2 */
  double bw_in;       /* effective bandwidth actor -> placement, > 0 */
  double bw_out;      /* tier 1 -> learner GPU, > 0 */
  double mem;         /* capacity of tier 1, >= 0 */
  double bw_out2;     /* tier 2 -> learner GPU (> 0 when tiers == 2) */
  double mem2;        /* capacity of tier 2 (tiers == 2) */
} edp_place_option;

/* Alg. 1 over opts[0..n): *best = index of the chosen placement, or n when
 * none is feasible (status EDP_ERR_EMPTY).  t_all (may be NULL) receives
 * T(p, x) for every option, +infinity for infeasible ones.
 * EDP_ERR_INVALID for NULL opts/best, n == 0, c_buf or x not finite and
 * > 0, or an option with a non-positive or non-finite bandwidth, a
 * negative capacity, or tiers not 1 or 2. */
EDP_API edp_status edp_place_choose(const edp_place_option *opts, uint32_t n,
                                    double c_buf, double x, uint32_t *best,
                                    double *t_all);

/* The placement map of Appendix D: the choice of edp_place_choose for each
 * per-sample size x[0..nx) (n where none is feasible), computed once so
 * that a change of x at run time is a lookup.  Errors as edp_place_choose;
 * an infeasible size is not an error here. */
EDP_API edp_status edp_place_map(const edp_place_option *opts, uint32_t n,
                                 double c_buf, const double *x, uint32_t nx,
                                 uint32_t *choice);

/* Effective bandwidths of this node's paths (Sec. 5.1: measured by
 * microbenchmarks on the deployment stack), in bytes moved per second;
 * each is the best of three timed transfers of `bytes`. */
typedef struct {
  double hbm_copy;       /* device -> device copy (each byte read and written) */
  double h2d_pinned;     /* cudaMemcpy, page-locked host -> device */
  double d2h_pinned;     /* cudaMemcpy, device -> page-locked host */
  double h2d_pageable;   /* cudaMemcpy, pageable host -> device */
  double zero_copy_read; /* a kernel reading page-locked host memory in place */
  double host_copy;      /* one CPU thread, memcpy pageable -> page-locked */
  double hbm_free;       /* free device memory (bytes) before the buffers below */
} edp_place_bw;

/* Measure edp_place_bw on `device` with buffers of `bytes` (a multiple of
 * 16, >= 1 MiB): allocates 2 x bytes of device memory, `bytes` of
 * page-locked and `bytes` of pageable host memory for the duration of the
 * call and frees them.  EDP_ERR_INVALID for bad arguments, EDP_ERR_OOM when
 * an allocation fails, EDP_ERR_CUDA for other CUDA errors.  Synchronises
 * the device. */
EDP_API edp_status edp_place_profile(int device, uint64_t bytes, edp_place_bw *out);

/* ABI version compiled into the library (EDP_ABI_VERSION). */
EDP_API int edp_abi_version(void);

#ifdef __cplusplus
}
#endif
#endif /* EDP_H */
