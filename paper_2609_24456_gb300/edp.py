"""Thin Python binding of libedp (C ABI declared in include/edp.h).

Argument marshalling only: every function forwards to the C entry point of the
same name, converting torch tensors to raw pointers and torch streams to
``cudaStream_t``.  PyTorch supplies device memory, page-locked host memory and
streams; every step of the data path runs in libedp's CUDA kernels.  There is
no fallback: if libedp.so cannot be loaded, every call raises.
"""
import ctypes as C
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libedp.so")

EDP_OK, EDP_ERR_INVALID, EDP_ERR_OOM, EDP_ERR_CUDA, EDP_ERR_TIMEOUT, \
    EDP_ERR_EMPTY, EDP_ERR_STATE = range(7)
STATUS_NAMES = ["EDP_OK", "EDP_ERR_INVALID", "EDP_ERR_OOM", "EDP_ERR_CUDA",
                "EDP_ERR_TIMEOUT", "EDP_ERR_EMPTY", "EDP_ERR_STATE"]
EDP_XFORM_STACK_F32, EDP_XFORM_HWC_CHW_BF16, EDP_XFORM_CHW_NORM_BF16 = range(3)
EDP_SAMPLE_UNIFORM, EDP_SAMPLE_PRIORITIZED, EDP_SAMPLE_PERMUTE = range(3)

ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_void_p, C.c_size_t)
FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p)


class edp_config(C.Structure):
    _fields_ = [("capacity", C.c_uint64), ("hbm_capacity", C.c_uint64),
                ("obs_c", C.c_uint32), ("obs_h", C.c_uint32),
                ("obs_w", C.c_uint32), ("transform", C.c_uint32),
                ("frame_stack", C.c_uint32), ("next_obs", C.c_uint32),
                ("tokens", C.c_uint32), ("prioritized", C.c_uint32),
                ("norm_mean", C.c_float * 4), ("norm_std", C.c_float * 4),
                ("alloc", ALLOC_FN), ("free", FREE_FN),
                ("alloc_user", C.c_void_p), ("device", C.c_int32),
                ("reserved", C.c_uint32 * 7)]


class edp_storage(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("tokens", C.c_void_p),
                ("host_obs", C.c_void_p), ("host_tokens", C.c_void_p),
                ("action", C.c_void_p), ("reward", C.c_void_p),
                ("done", C.c_void_p)]


class edp_fields(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("tokens", C.c_void_p),
                ("action", C.c_void_p), ("reward", C.c_void_p),
                ("done", C.c_void_p)]


class edp_batch(C.Structure):
    _fields_ = [("obs", C.c_void_p), ("next_obs", C.c_void_p),
                ("action", C.c_void_p), ("reward", C.c_void_p),
                ("done", C.c_void_p), ("tokens", C.c_void_p),
                ("q", C.c_void_p), ("isw", C.c_void_p), ("beta", C.c_double),
                ("gather_src", C.c_void_p * 2), ("gather_dst", C.c_void_p * 2)]


class edp_info(C.Structure):
    _fields_ = [("capacity", C.c_uint64), ("hbm_capacity", C.c_uint64),
                ("total", C.c_uint64), ("size", C.c_uint64),
                ("head", C.c_uint64), ("oldest", C.c_uint64),
                ("n_valid", C.c_uint64), ("tree_depth", C.c_uint32),
                ("tree_fanout", C.c_uint32), ("tree_leaves", C.c_void_p),
                ("tree_level", C.c_void_p * 8), ("pending_q", C.c_void_p),
                ("max_q", C.c_void_p), ("norm_path", C.c_uint32)]


class edp_sched_costs(C.Structure):
    _fields_ = [("t_rollout", C.c_double), ("t_update", C.c_double),
                ("t_sync_ing", C.c_double), ("t_sync_del", C.c_double),
                ("n_ing", C.c_uint32), ("n_del", C.c_uint32),
                ("g_ing", C.POINTER(C.c_double)), ("t_ing", C.POINTER(C.c_double)),
                ("g_del", C.POINTER(C.c_double)), ("t_del", C.POINTER(C.c_double)),
                ("contention_ing", C.c_double), ("contention_del", C.c_double)]


class edp_sched_choice(C.Structure):
    _fields_ = [("overlap_ing", C.c_uint32), ("overlap_del", C.c_uint32),
                ("i_ing", C.c_uint32), ("i_del", C.c_uint32),
                ("g_ing", C.c_double), ("g_del", C.c_double),
                ("t_ing_path", C.c_double), ("t_del_path", C.c_double),
                ("t_iter", C.c_double)]


EDP_PLACE_HOST_PAGEABLE, EDP_PLACE_HOST_PINNED, EDP_PLACE_GPU, EDP_PLACE_GPU_HOST = range(4)


class edp_place_option(C.Structure):
    _fields_ = [("kind", C.c_uint32), ("tiers", C.c_uint32), ("bw_in", C.c_double),
                ("bw_out", C.c_double), ("mem", C.c_double), ("bw_out2", C.c_double),
                ("mem2", C.c_double)]


class edp_place_bw(C.Structure):
    _fields_ = [("hbm_copy", C.c_double), ("h2d_pinned", C.c_double),
                ("d2h_pinned", C.c_double), ("h2d_pageable", C.c_double),
                ("zero_copy_read", C.c_double), ("host_copy", C.c_double),
                ("hbm_free", C.c_double)]


# exported symbols and their signatures (restype, argtypes)
_VP, _U32, _U64, _D = C.c_void_p, C.c_uint32, C.c_uint64, C.c_double
SIGNATURES = {
    "edp_create": (C.c_int, [C.POINTER(edp_config), C.POINTER(edp_storage),
                             C.POINTER(C.c_void_p)]),
    "edp_destroy": (C.c_int, [_VP]),
    "edp_ingest": (C.c_int, [_VP, C.POINTER(edp_fields), _U64, _VP, _VP]),
    "edp_sample": (C.c_int, [_VP, C.c_int, _U32, _U64, _U64, _VP, _VP, _VP]),
    "edp_deliver": (C.c_int, [_VP, _VP, _U32, C.POINTER(edp_batch), _VP]),
    "edp_sample_deliver": (C.c_int, [_VP, _U32, _U64, _U64, _VP, C.POINTER(edp_batch), _VP]),
    "edp_update_priorities": (C.c_int, [_VP, _VP, _VP, _U32, _VP]),
    "edp_update_priorities_td": (C.c_int, [_VP, _VP, _VP, _U32, _D, _D, _VP]),
    "edp_update_priorities_td_static": (C.c_int, [_VP, _VP, _VP, _U32, _D, _D, _VP]),
    "edp_priorities_from_td": (C.c_int, [_VP, _VP, _U32, _D, _D, _VP, _VP]),
    "edp_gae": (C.c_int, [_VP, _VP, _VP, _VP, _U32, _U32, _D, _D, _VP, _VP,
                          _VP, _VP]),
    "edp_tree_total": (C.c_int, [_VP, _VP, _VP]),
    "edp_route_prioritized": (C.c_int, [_VP, _VP, _U32, _U32, _U32, _U32, _U64, _U64,
                                        _VP, _VP, _VP]),
    "edp_sample_targets": (C.c_int, [_VP, _VP, _U32, _VP, _VP, _VP]),
    "edp_batch_qmin": (C.c_int, [_VP, _VP, _U32, _VP, _VP]),
    "edp_is_weights": (C.c_int, [_VP, _VP, _U32, _VP, _D, _VP, _VP]),
    "edp_gae_stats": (C.c_int, [_VP, _VP, _VP, _VP, _U32, _U32, _D, _D, _VP, _VP, _VP,
                                _VP]),
    "edp_gae_normalize": (C.c_int, [_VP, _VP, _U64, _VP, _VP, _VP]),
    "edp_get_counters": (C.c_int, [_VP, _VP]),
    "edp_reset_counters": (C.c_int, [_VP]),
    "edp_sync": (C.c_int, [_VP, _VP]),
    "edp_last_error": (C.c_char_p, [_VP]),
    "edp_get_info": (C.c_int, [_VP, C.POINTER(edp_info)]),
    "edp_probe_host_read": (C.c_int, [_VP, _U64, _VP, _VP]),
    "edp_abi_version": (C.c_int, []),
    "edp_sched_choose": (C.c_int, [C.POINTER(edp_sched_costs),
                                   C.POINTER(edp_sched_choice), _VP]),
    "edp_sched_granularities": (_U32, [_U32, _U32, _VP, _U32]),
    "edp_place_choose": (C.c_int, [C.POINTER(edp_place_option), _U32, _D, _D,
                                   C.POINTER(C.c_uint32), _VP]),
    "edp_place_map": (C.c_int, [C.POINTER(edp_place_option), _U32, _D, _VP, _U32, _VP]),
    "edp_place_profile": (C.c_int, [C.c_int, _U64, C.POINTER(edp_place_bw)]),
    "edp_migrate": (C.c_int, [_VP, _VP, _VP]),
    "edp_save": (C.c_int, [_VP, C.c_char_p, _VP]),
    "edp_load": (C.c_int, [_VP, C.c_char_p, _VP]),
    "edp_grpo_advantage": (C.c_int, [_VP, _VP, _VP, _U32, C.c_float, _VP, _VP]),
    "edp_pack_deliver": (C.c_int, [_VP, _VP, _VP, _U64, _VP, _U32, _VP, _VP, _VP, _VP,
                                   _U64, _VP]),
    "edp_grpo_pack_deliver": (C.c_int, [_VP, _VP, _VP, _U32, C.c_float, _VP, _VP, _VP, _U64,
                                        _VP, _U32, _VP, _VP, _VP, _U64, _VP]),
}

_lib = None


def lib():
    """Load libedp.so (raises if it is missing: there is no fallback)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                "libedp.so not built (%s); run paper_2609_24456_gb300.build.build()"
                % LIB_PATH)
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


class EdpError(RuntimeError):
    def __init__(self, status, msg):
        self.status = status
        name = STATUS_NAMES[status] if 0 <= status < len(STATUS_NAMES) else str(status)
        super().__init__("%s: %s" % (name, msg))


def ptr(x):
    """Raw address of a tensor / int / None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return x.data_ptr()


def stream_handle(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(ctx, status, what):
    if status != EDP_OK:
        msg = lib().edp_last_error(ctx) if ctx else b""
        raise EdpError(status, "%s: %s" % (what, (msg or b"").decode()))
    return status


# --- the C entry points -------------------------------------------------------
def edp_create(cfg: edp_config, st: edp_storage) -> int:
    out = C.c_void_p()
    s = lib().edp_create(C.byref(cfg), C.byref(st), C.byref(out))
    if s != EDP_OK:
        raise EdpError(s, "edp_create failed (details on stderr)")
    return out.value


def edp_destroy(ctx):
    return _check(None, lib().edp_destroy(ctx), "edp_destroy")


def edp_ingest(ctx, obs, n, tokens=None, action=None, reward=None, done=None,
               q=None, stream=None):
    f = edp_fields(ptr(obs), ptr(tokens), ptr(action), ptr(reward), ptr(done))
    return _check(ctx, lib().edp_ingest(ctx, C.byref(f), n, ptr(q),
                                        stream_handle(stream)), "edp_ingest")


def edp_sample(ctx, mode, batch, seed, round_, idx, q=None, stream=None):
    return _check(ctx, lib().edp_sample(ctx, mode, batch, seed, round_, ptr(idx),
                                        ptr(q), stream_handle(stream)),
                  "edp_sample")


def make_batch(obs, next_obs=None, action=None, reward=None, done=None,
               tokens=None, q=None, isw=None, beta=0.0, gather=()):
    b = edp_batch()
    b.obs, b.next_obs = ptr(obs), ptr(next_obs)
    b.action, b.reward, b.done = ptr(action), ptr(reward), ptr(done)
    b.tokens, b.q, b.isw, b.beta = ptr(tokens), ptr(q), ptr(isw), float(beta)
    for i, (src, dst) in enumerate(gather):
        b.gather_src[i] = ptr(src)
        b.gather_dst[i] = ptr(dst)
    return b


def edp_sample_deliver(ctx, batch, seed, round_, idx, out: edp_batch, stream=None):
    return _check(ctx, lib().edp_sample_deliver(ctx, batch, seed, round_, ptr(idx),
                                                C.byref(out), stream_handle(stream)),
                  "edp_sample_deliver")


def edp_deliver(ctx, idx, batch, out: edp_batch, stream=None):
    return _check(ctx, lib().edp_deliver(ctx, ptr(idx), batch, C.byref(out),
                                         stream_handle(stream)), "edp_deliver")


def edp_update_priorities(ctx, idx, q, n, stream=None):
    return _check(ctx, lib().edp_update_priorities(ctx, ptr(idx), ptr(q), n,
                                                   stream_handle(stream)),
                  "edp_update_priorities")


def edp_update_priorities_td(ctx, idx, td, n, alpha, eps, stream=None):
    return _check(ctx, lib().edp_update_priorities_td(
        ctx, ptr(idx), ptr(td), n, alpha, eps, stream_handle(stream)),
        "edp_update_priorities_td")


def edp_update_priorities_td_static(ctx, idx, td, n, alpha, eps, stream=None):
    """Allocation-free edp_update_priorities_td (fixed per-device scratch of
    16384 pairs; see include/edp.h)."""
    return _check(ctx, lib().edp_update_priorities_td_static(
        ctx, ptr(idx), ptr(td), n, alpha, eps, stream_handle(stream)),
        "edp_update_priorities_td_static")


def edp_priorities_from_td(ctx, td, n, alpha, eps, q, stream=None):
    return _check(ctx, lib().edp_priorities_from_td(
        ctx, ptr(td), n, alpha, eps, ptr(q), stream_handle(stream)),
        "edp_priorities_from_td")


def edp_gae(ctx, r, v, d, T, E, gamma, lam, adv=None, ret=None, adv_norm=None,
            stream=None):
    return _check(ctx, lib().edp_gae(ctx, ptr(r), ptr(v), ptr(d), T, E, gamma,
                                     lam, ptr(adv), ptr(ret), ptr(adv_norm),
                                     stream_handle(stream)), "edp_gae")


# --- sharded buffer (include/edp.h, "Sharded buffer") ---------------------------
def edp_tree_total(ctx, total, stream=None):
    return _check(ctx, lib().edp_tree_total(ctx, ptr(total), stream_handle(stream)),
                  "edp_tree_total")


def edp_route_prioritized(ctx, totals, G, batch, k0, n, seed, round_, local_t, counts,
                          stream=None):
    return _check(ctx, lib().edp_route_prioritized(
        ctx, ptr(totals), G, batch, k0, n, seed, round_, ptr(local_t), ptr(counts),
        stream_handle(stream)), "edp_route_prioritized")


def edp_sample_targets(ctx, targets, n, idx, q=None, stream=None):
    return _check(ctx, lib().edp_sample_targets(ctx, ptr(targets), n, ptr(idx), ptr(q),
                                                stream_handle(stream)), "edp_sample_targets")


def edp_batch_qmin(ctx, q, n, qmin, stream=None):
    return _check(ctx, lib().edp_batch_qmin(ctx, ptr(q), n, ptr(qmin),
                                            stream_handle(stream)), "edp_batch_qmin")


def edp_is_weights(ctx, q, n, qmin, beta, w, stream=None):
    return _check(ctx, lib().edp_is_weights(ctx, ptr(q), n, ptr(qmin), beta, ptr(w),
                                            stream_handle(stream)), "edp_is_weights")


def edp_gae_stats(ctx, r, v, d, T, E, gamma, lam, adv, stats, ret=None, stream=None):
    return _check(ctx, lib().edp_gae_stats(ctx, ptr(r), ptr(v), ptr(d), T, E, gamma, lam,
                                           ptr(adv), ptr(ret), ptr(stats),
                                           stream_handle(stream)), "edp_gae_stats")


def edp_gae_normalize(ctx, adv, n, stats, adv_norm, stream=None):
    return _check(ctx, lib().edp_gae_normalize(ctx, ptr(adv), n, ptr(stats), ptr(adv_norm),
                                               stream_handle(stream)), "edp_gae_normalize")


class edp_counters(C.Structure):
    _fields_ = [("calls", _U64), ("ingested", _U64), ("sampled", _U64), ("delivered", _U64),
                ("hbm_read", _U64), ("hbm_write", _U64), ("link_read", _U64),
                ("link_write", _U64)]


def edp_get_counters(ctx) -> dict:
    out = edp_counters()
    _check(ctx, lib().edp_get_counters(ctx, C.byref(out)), "edp_get_counters")
    return {name: getattr(out, name) for name, _ in edp_counters._fields_}


def edp_reset_counters(ctx):
    return _check(ctx, lib().edp_reset_counters(ctx), "edp_reset_counters")


def edp_sync(ctx, stream=None):
    return _check(ctx, lib().edp_sync(ctx, stream_handle(stream)), "edp_sync")


def edp_sync_status(ctx, stream=None):
    """edp_sync returning (status, message) instead of raising."""
    s = lib().edp_sync(ctx, stream_handle(stream))
    return s, (lib().edp_last_error(ctx) or b"").decode()


def edp_last_error(ctx):
    return (lib().edp_last_error(ctx) or b"").decode()


def edp_get_info(ctx) -> edp_info:
    out = edp_info()
    _check(ctx, lib().edp_get_info(ctx, C.byref(out)), "edp_get_info")
    return out


def edp_probe_host_read(host_src, nbytes, d_fold, stream=None):
    s = lib().edp_probe_host_read(ptr(host_src), nbytes, ptr(d_fold),
                                  stream_handle(stream))
    if s != EDP_OK:
        raise EdpError(s, "edp_probe_host_read")


def edp_abi_version():
    return lib().edp_abi_version()


# --- storage plumbing (torch allocations) -------------------------------------
def make_config(capacity, obs_shape, transform, hbm_capacity=None,
                frame_stack=1, next_obs=False, tokens=0, prioritized=False,
                norm_mean=(0.0,) * 4, norm_std=(1.0,) * 4, device=0):
    """obs_shape = (c, h, w) of the stored observation."""
    cfg = edp_config()
    cfg.capacity = capacity
    cfg.hbm_capacity = capacity if hbm_capacity is None else hbm_capacity
    cfg.obs_c, cfg.obs_h, cfg.obs_w = obs_shape
    cfg.transform = transform
    cfg.frame_stack = frame_stack
    cfg.next_obs = int(bool(next_obs))
    cfg.tokens = tokens
    cfg.prioritized = int(bool(prioritized))
    for i in range(4):
        cfg.norm_mean[i] = list(norm_mean)[i] if i < len(norm_mean) else 0.0
        cfg.norm_std[i] = list(norm_std)[i] if i < len(norm_std) else 1.0
    cfg.device = device
    return cfg


class Ring:
    """Caller-side storage of a ring plus its context handle.

    Tensors are allocated with torch (device memory for HBM fields,
    pin_memory for the host tier) and handed to edp_create as raw pointers.
    """

    def __init__(self, cfg: edp_config, action=True, reward=True, done=True):
        import torch
        self.cfg = cfg
        dev = torch.device("cuda", cfg.device)
        ob = cfg.obs_c * cfg.obs_h * cfg.obs_w
        cap, cap_h = cfg.capacity, cfg.hbm_capacity
        self.obs = torch.empty((cap_h, ob), dtype=torch.uint8, device=dev)
        self.tokens = (torch.empty((cap_h, cfg.tokens), dtype=torch.int32,
                                   device=dev) if cfg.tokens else None)
        self.host_obs = self.host_tokens = None
        if cap_h < cap:
            self.host_obs = torch.empty((cap - cap_h, ob), dtype=torch.uint8,
                                        pin_memory=True)
            if cfg.tokens:
                self.host_tokens = torch.empty((cap - cap_h, cfg.tokens),
                                               dtype=torch.int32,
                                               pin_memory=True)
        self.action = torch.zeros(cap, dtype=torch.int32, device=dev) if action else None
        self.reward = torch.zeros(cap, dtype=torch.float32, device=dev) if reward else None
        self.done = torch.zeros(cap, dtype=torch.uint8, device=dev) if done else None
        st = edp_storage(ptr(self.obs), ptr(self.tokens), ptr(self.host_obs),
                         ptr(self.host_tokens), ptr(self.action),
                         ptr(self.reward), ptr(self.done))
        self.ctx = edp_create(cfg, st)

    def info(self):
        return edp_get_info(self.ctx)

    def close(self):
        if self.ctx:
            edp_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def _dvec(xs):
    return (C.c_double * len(xs))(*[float(x) for x in xs])


def edp_sched_choose(t_rollout, t_update, t_sync_ing, t_sync_del, g_ing, t_ing,
                     g_del, t_del, all_scores=False, contention_ing=0.0,
                     contention_del=0.0):
    """Latency-minimising timing and granularity (host only).  Returns the
    edp_sched_choice, and with all_scores the [2][2][n_ing][n_del] list of
    every candidate's T_iter."""
    gi, ti, gd, td = _dvec(g_ing), _dvec(t_ing), _dvec(g_del), _dvec(t_del)
    c = edp_sched_costs(t_rollout, t_update, t_sync_ing, t_sync_del, len(g_ing),
                        len(g_del), gi, ti, gd, td, contention_ing, contention_del)
    out = edp_sched_choice()
    n = 4 * len(g_ing) * len(g_del)
    buf = (C.c_double * n)() if all_scores else None
    st = lib().edp_sched_choose(C.byref(c), C.byref(out),
                                C.cast(buf, C.c_void_p) if buf is not None else None)
    if st != EDP_OK:
        raise EdpError(st, "edp_sched_choose: invalid costs")
    return (out, list(buf)) if all_scores else out


def edp_sched_granularities(on_policy, m):
    """Candidate granularities for an off- or on-policy configuration."""
    n = lib().edp_sched_granularities(int(bool(on_policy)), m, None, 0)
    buf = (C.c_double * max(n, 1))()
    lib().edp_sched_granularities(int(bool(on_policy)), m, C.cast(buf, C.c_void_p), n)
    return list(buf)[:n]


def _options(opts):
    """opts: sequence of dicts with kind, bw_in, bw_out, mem and, for two
    tiers, bw_out2 and mem2."""
    arr = (edp_place_option * len(opts))()
    for a, o in zip(arr, opts):
        two = "bw_out2" in o
        a.kind, a.tiers = o.get("kind", 0), 2 if two else 1
        a.bw_in, a.bw_out, a.mem = o["bw_in"], o["bw_out"], o["mem"]
        a.bw_out2, a.mem2 = (o["bw_out2"], o["mem2"]) if two else (0.0, 0.0)
    return arr


def edp_place_choose(opts, c_buf, x):
    """(index of the chosen placement or len(opts) if none fits, [T(p, x)])."""
    arr = _options(opts)
    best = C.c_uint32()
    t = (C.c_double * len(opts))()
    st = lib().edp_place_choose(arr, len(opts), float(c_buf), float(x), C.byref(best),
                                C.cast(t, C.c_void_p))
    if st not in (EDP_OK, EDP_ERR_EMPTY):
        raise EdpError(st, "edp_place_choose: invalid options")
    return best.value, list(t)


def edp_place_map(opts, c_buf, xs):
    """The placement chosen for every per-sample size in xs."""
    arr = _options(opts)
    xv = _dvec(xs)
    out = (C.c_uint32 * max(len(xs), 1))()
    st = lib().edp_place_map(arr, len(opts), float(c_buf), C.cast(xv, C.c_void_p),
                             len(xs), C.cast(out, C.c_void_p))
    if st != EDP_OK:
        raise EdpError(st, "edp_place_map: invalid options")
    return list(out)[:len(xs)]


def edp_place_profile(device=0, nbytes=1 << 30):
    """Effective bandwidths of this node's paths (bytes/s) as a dict."""
    out = edp_place_bw()
    st = lib().edp_place_profile(int(device), int(nbytes), C.byref(out))
    if st != EDP_OK:
        raise EdpError(st, "edp_place_profile failed (status %d)" % st)
    return {f: getattr(out, f) for f, _ in edp_place_bw._fields_}


def edp_migrate(src_ctx, dst_ctx, stream=None):
    """Move src's experience state into the empty context dst (new placement)."""
    return _check(dst_ctx, lib().edp_migrate(src_ctx, dst_ctx, stream_handle(stream)),
                  "edp_migrate")


def edp_grpo_advantage(ctx, r, group_off, n_groups, eps, adv, stream=None):
    return _check(ctx, lib().edp_grpo_advantage(ctx, ptr(r), ptr(group_off), n_groups,
                                                float(eps), ptr(adv), stream_handle(stream)),
                  "edp_grpo_advantage")


def edp_pack_deliver(ctx, tokens, seq_off, n_seq, idx, batch, out_tokens, out_off,
                     out_cap, seq_value=None, out_value=None, stream=None):
    return _check(ctx, lib().edp_pack_deliver(
        ctx, ptr(tokens), ptr(seq_off), n_seq, ptr(idx), batch, ptr(seq_value),
        ptr(out_tokens), ptr(out_off), ptr(out_value), out_cap, stream_handle(stream)),
        "edp_pack_deliver")


def edp_grpo_pack_deliver(ctx, r, group_off, n_groups, eps, adv, tokens, seq_off, n_seq,
                          idx, batch, out_tokens, out_off, out_cap, out_value=None,
                          stream=None):
    return _check(ctx, lib().edp_grpo_pack_deliver(
        ctx, ptr(r), ptr(group_off), n_groups, eps, ptr(adv), ptr(tokens), ptr(seq_off),
        n_seq, ptr(idx), batch, ptr(out_tokens), ptr(out_off), ptr(out_value), out_cap,
        stream_handle(stream)), "edp_grpo_pack_deliver")


def edp_save(ctx, path, stream=None):
    """Write the context's retained experience to the file `path`."""
    return _check(ctx, lib().edp_save(ctx, os.fsencode(path), stream_handle(stream)),
                  "edp_save")


def edp_load(ctx, path, stream=None):
    """Read a checkpoint written by edp_save into the empty context."""
    return _check(ctx, lib().edp_load(ctx, os.fsencode(path), stream_handle(stream)),
                  "edp_load")
