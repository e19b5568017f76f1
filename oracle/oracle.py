"""ctypes/numpy front end of the plain-C oracle (test infrastructure only).

Each wrapper names the method it follows; the arithmetic lives in
``edp_oracle.c`` and is documented there.
"""
import ctypes as C

import numpy as np

from . import build as _build

__all__ = [
    "lib", "philox4x32_10", "philox_u64", "mulhi64", "ring_size", "ring_slot",
    "ring_offset", "ring_write", "ingest_leaves", "update_leaves", "leaf_sum",
    "priorities_from_td", "sample_uniform", "stratum_target",
    "ingest_leaves_default",
    "sample_prioritized_scan", "sample_prioritized_bisect", "is_weights",
    "unit_f32", "bf16_rne", "norm_bf16", "dqn_stack", "deliver_dqn",
    "hwc_to_chw_bf16", "deliver_ppo", "norm_chw_bf16", "deliver_mm", "gae",
    "normalize", "permutation", "tier_of", "PerState",
]

_lib = None


def lib():
    global _lib
    if _lib is None:
        path = _build.build()
        L = C.CDLL(path)
        u8p = C.POINTER(C.c_uint8)
        u16p = C.POINTER(C.c_uint16)
        u32p = C.POINTER(C.c_uint32)
        i32p = C.POINTER(C.c_int32)
        i64p = C.POINTER(C.c_int64)
        f32p = C.POINTER(C.c_float)
        f64p = C.POINTER(C.c_double)
        u64, u32 = C.c_uint64, C.c_uint32
        sig = {
            "orc_philox4x32_10": (None, [u32p, u32p, u32p]),
            "orc_philox_u64": (u64, [u64, u32, u64, u32]),
            "orc_mulhi64": (u64, [u64, u64]),
            "orc_ring_size": (u64, [u64, u64]),
            "orc_ring_slot": (u64, [u64, u64, u64]),
            "orc_ring_offset": (u64, [u64, u64, u64]),
            "orc_ring_write": (None, [u8p, u64, u64, u64, u8p, u64]),
            "orc_ingest_leaves": (None, [u32p, u64, u64, C.c_int, u32p, u64,
                                         u32p, u32p]),
            "orc_update_leaves": (None, [u32p, u64, u64, C.c_int, i64p, u32p,
                                         u64, u32p, u32p]),
            "orc_leaf_sum": (u64, [u32p, u64, u64]),
            "orc_priority_from_td": (u32, [C.c_double, C.c_double, C.c_double]),
            "orc_priorities_from_td": (None, [f32p, u64, C.c_double,
                                              C.c_double, u32p]),
            "orc_sample_uniform": (None, [u64, u64, u64, u32, u64, u64, i64p]),
            "orc_stratum_target": (u64, [u64, u32, u32, u64]),
            "orc_sample_prioritized_scan": (C.c_int, [u32p, u64, u32, u64, u64,
                                                      i64p, u32p]),
            "orc_sample_prioritized_bisect": (C.c_int, [u32p, u64, u32, u64,
                                                        u64, i64p, u32p]),
            "orc_is_weights": (None, [u32p, u32, C.c_double, f32p]),
            "orc_unit_f32": (C.c_float, [C.c_uint8]),
            "orc_bf16_rne": (C.c_uint16, [C.c_float]),
            "orc_norm_bf16": (C.c_uint16, [C.c_uint8, C.c_float, C.c_float]),
            "orc_dqn_stack": (None, [u8p, u8p, u64, u64, u32, u32, C.c_int64,
                                     f32p, f32p]),
            "orc_deliver_dqn": (None, [u8p, u8p, i32p, f32p, u64, u64, u32, u32,
                                       i64p, u32, f32p, f32p, i32p, f32p, u8p]),
            "orc_hwc_to_chw_bf16": (None, [u8p, u32, u32, u32, u16p]),
            "orc_deliver_ppo": (None, [u8p, u64, u64, u32, u32, u32, i64p, u32,
                                       f32p, f32p, u16p, f32p, f32p]),
            "orc_norm_chw_bf16": (None, [u8p, u32, u64, f32p, f32p, u16p]),
            "orc_deliver_mm": (None, [u8p, i32p, f32p, u32, u64, u32, i64p, u32,
                                      f32p, f32p, u16p, i32p, f32p]),
            "orc_gae": (None, [f32p, f32p, u8p, u32, u32, C.c_double,
                               C.c_double, f64p, f64p]),
            "orc_normalize": (None, [f64p, u64, f64p, f64p, f64p]),
            "orc_permutation": (C.c_int, [u32, u64, u64, i64p]),
            "orc_tier_of": (None, [u64, u64, u64, u64, i32p,
                                   C.POINTER(C.c_uint64)]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _p(a, ctype):
    if a is None:
        return None
    return a.ctypes.data_as(C.POINTER(ctype))


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a


# -- Philox (Salmon et al. SC'11) ------------------------------------------
def philox4x32_10(ctr, key):
    c = _c(ctr, np.uint32)
    k = _c(key, np.uint32)
    o = np.zeros(4, np.uint32)
    lib().orc_philox4x32_10(_p(c, C.c_uint32), _p(k, C.c_uint32),
                            _p(o, C.c_uint32))
    return o


def philox_u64(seed, j, round_, stream):
    return int(lib().orc_philox_u64(seed, j, round_, stream))


def mulhi64(a, n):
    return int(lib().orc_mulhi64(a, n))


# -- ring ------------------------------------------------------------------
def ring_size(cap, total):
    return int(lib().orc_ring_size(cap, total))


def ring_slot(cap, total, k):
    return int(lib().orc_ring_slot(cap, total, k))


def ring_offset(cap, total, slot):
    return int(lib().orc_ring_offset(cap, total, slot))


def ring_write(ring, cap, total, src):
    """Insert src[n, ...] into ring[cap, ...] at logical ids total.. (FIFO)."""
    assert ring.flags.c_contiguous and src.flags.c_contiguous
    assert ring.dtype == src.dtype
    rec = ring.nbytes // cap
    n = src.shape[0]
    lib().orc_ring_write(ring.ctypes.data_as(C.POINTER(C.c_uint8)), cap, rec,
                         total, src.ctypes.data_as(C.POINTER(C.c_uint8)), n)


class PerState:
    """Leaves of the priority distribution plus the deferred priority and the
    running maximum (PER, Schaul et al.)."""

    def __init__(self, cap, defer):
        self.cap = cap
        self.defer = int(bool(defer))
        self.leaves = np.zeros(cap, np.uint32)
        self.pending = np.zeros(1, np.uint32)
        self.qmax = np.array([1 << 20], np.uint32)


def ingest_leaves(st, total, q):
    n = 0 if q is None else len(q)
    qq = None if q is None else _c(q, np.uint32)
    lib().orc_ingest_leaves(_p(st.leaves, C.c_uint32), st.cap, total, st.defer,
                            _p(qq, C.c_uint32), n, _p(st.pending, C.c_uint32),
                            _p(st.qmax, C.c_uint32))


def ingest_leaves_default(st, total, n):
    lib().orc_ingest_leaves(_p(st.leaves, C.c_uint32), st.cap, total, st.defer,
                            None, n, _p(st.pending, C.c_uint32),
                            _p(st.qmax, C.c_uint32))


def update_leaves(st, total, idx, q):
    i = _c(idx, np.int64)
    qq = _c(q, np.uint32)
    lib().orc_update_leaves(_p(st.leaves, C.c_uint32), st.cap, total, st.defer,
                            _p(i, C.c_int64), _p(qq, C.c_uint32), len(i),
                            _p(st.pending, C.c_uint32), _p(st.qmax, C.c_uint32))


def leaf_sum(leaves, lo, hi):
    leaves = _c(leaves, np.uint32)
    return int(lib().orc_leaf_sum(_p(leaves, C.c_uint32), lo, hi))


def priorities_from_td(td, alpha, eps):
    td = _c(td, np.float32)
    q = np.zeros(len(td), np.uint32)
    lib().orc_priorities_from_td(_p(td, C.c_float), len(td), alpha, eps,
                                 _p(q, C.c_uint32))
    return q


# -- samplers ----------------------------------------------------------------
def sample_uniform(cap, total, n_valid, B, seed, round_):
    idx = np.zeros(B, np.int64)
    lib().orc_sample_uniform(cap, total, n_valid, B, seed, round_,
                             _p(idx, C.c_int64))
    return idx


def stratum_target(S, B, k, u):
    return int(lib().orc_stratum_target(S, B, k, u))


def _prio(fn, leaves, B, seed, round_):
    leaves = _c(leaves, np.uint32)
    idx = np.zeros(B, np.int64)
    q = np.zeros(B, np.uint32)
    rc = fn(_p(leaves, C.c_uint32), len(leaves), B, seed, round_,
            _p(idx, C.c_int64), _p(q, C.c_uint32))
    if rc != 0:
        raise ValueError("total priority is zero")
    return idx, q


def sample_prioritized_scan(leaves, B, seed, round_):
    return _prio(lib().orc_sample_prioritized_scan, leaves, B, seed, round_)


def sample_prioritized_bisect(leaves, B, seed, round_):
    return _prio(lib().orc_sample_prioritized_bisect, leaves, B, seed, round_)


def is_weights(q, beta):
    q = _c(q, np.uint32)
    w = np.zeros(len(q), np.float32)
    lib().orc_is_weights(_p(q, C.c_uint32), len(q), beta, _p(w, C.c_float))
    return w


# -- transforms ----------------------------------------------------------------
def unit_f32(b):
    return np.float32(lib().orc_unit_f32(int(b)))


def bf16_rne(x):
    return int(lib().orc_bf16_rne(float(np.float32(x))))


def norm_bf16(b, mean, std):
    return int(lib().orc_norm_bf16(int(b), float(np.float32(mean)),
                                   float(np.float32(std))))


# -- deliveries ------------------------------------------------------------------
def dqn_stack(frames, done, cap, total, K, slot, with_next=True):
    F = frames.shape[1]
    obs = np.zeros((K, F), np.float32)
    nxt = np.zeros((K, F), np.float32) if with_next else None
    lib().orc_dqn_stack(_p(frames, C.c_uint8), _p(done, C.c_uint8), cap, total,
                        F, K, int(slot), _p(obs, C.c_float), _p(nxt, C.c_float))
    return obs, nxt


def deliver_dqn(frames, done, action, reward, cap, total, K, idx,
                with_next=True):
    """frames [cap, F] uint8 (any array with that buffer layout)."""
    F = frames.shape[1]
    idx = _c(idx, np.int64)
    B = len(idx)
    obs = np.zeros((B, K, F), np.float32)
    nxt = np.zeros((B, K, F), np.float32) if with_next else None
    act = np.zeros(B, np.int32)
    rew = np.zeros(B, np.float32)
    dn = np.zeros(B, np.uint8)
    lib().orc_deliver_dqn(_p(frames, C.c_uint8), _p(done, C.c_uint8),
                          _p(action, C.c_int32), _p(reward, C.c_float), cap,
                          total, F, K, _p(idx, C.c_int64), B, _p(obs, C.c_float),
                          _p(nxt, C.c_float), _p(act, C.c_int32),
                          _p(rew, C.c_float), _p(dn, C.c_uint8))
    return obs, nxt, act, rew, dn


def hwc_to_chw_bf16(hwc):
    H, W, Cc = hwc.shape
    hwc = _c(hwc, np.uint8)
    out = np.zeros((Cc, H, W), np.uint16)
    lib().orc_hwc_to_chw_bf16(_p(hwc, C.c_uint8), H, W, Cc,
                              _p(out, C.c_uint16))
    return out


def deliver_ppo(obs_ring, cap, total, H, W, Cc, idx, adv, ret):
    idx = _c(idx, np.int64)
    B = len(idx)
    out = np.zeros((B, Cc, H, W), np.uint16)
    a = np.zeros(B, np.float32)
    r = np.zeros(B, np.float32)
    adv = _c(adv, np.float32)
    ret = _c(ret, np.float32)
    lib().orc_deliver_ppo(_p(obs_ring, C.c_uint8), cap, total, H, W, Cc,
                          _p(idx, C.c_int64), B, _p(adv, C.c_float),
                          _p(ret, C.c_float), _p(out, C.c_uint16),
                          _p(a, C.c_float), _p(r, C.c_float))
    return out, a, r


def norm_chw_bf16(chw, mean, std):
    Cc = chw.shape[0]
    HW = chw.size // Cc
    chw = _c(chw, np.uint8)
    m = _c(mean, np.float32)
    s = _c(std, np.float32)
    out = np.zeros(chw.shape, np.uint16)
    lib().orc_norm_chw_bf16(_p(chw, C.c_uint8), Cc, HW, _p(m, C.c_float),
                            _p(s, C.c_float), _p(out, C.c_uint16))
    return out


def deliver_mm(obs_ring, tok_ring, reward, Cc, HW, idx, mean, std):
    idx = _c(idx, np.int64)
    B = len(idx)
    L = tok_ring.shape[1] if tok_ring is not None else 0
    out = np.zeros((B, Cc * HW), np.uint16)
    tok = np.zeros((B, L), np.int32)
    rew = np.zeros(B, np.float32)
    m = _c(mean, np.float32)
    s = _c(std, np.float32)
    lib().orc_deliver_mm(_p(obs_ring, C.c_uint8), _p(tok_ring, C.c_int32),
                         _p(reward, C.c_float), Cc, HW, L, _p(idx, C.c_int64),
                         B, _p(m, C.c_float), _p(s, C.c_float),
                         _p(out, C.c_uint16), _p(tok, C.c_int32),
                         _p(rew, C.c_float))
    return out, tok, rew


# -- GAE (Schulman et al.) -------------------------------------------------------
def gae(r, v, d, gamma, lam):
    r = _c(r, np.float32)
    v = _c(v, np.float32)
    d = _c(d, np.uint8)
    T, E = r.shape
    assert v.shape == (T + 1, E) and d.shape == (T, E)
    adv = np.zeros((T, E), np.float64)
    ret = np.zeros((T, E), np.float64)
    lib().orc_gae(_p(r, C.c_float), _p(v, C.c_float), _p(d, C.c_uint8), T, E,
                  gamma, lam, _p(adv, C.c_double), _p(ret, C.c_double))
    return adv, ret


def normalize(a):
    a = _c(a, np.float64)
    out = np.zeros_like(a)
    m = np.zeros(1)
    s = np.zeros(1)
    lib().orc_normalize(_p(a, C.c_double), a.size, _p(out, C.c_double),
                        _p(m, C.c_double), _p(s, C.c_double))
    return out, float(m[0]), float(s[0])


def permutation(n, seed, iteration):
    perm = np.zeros(n, np.int64)
    rc = lib().orc_permutation(n, seed, iteration, _p(perm, C.c_int64))
    if rc != 0:
        raise MemoryError
    return perm


def tier_of(cap, cap_h, total, L):
    t = C.c_int32()
    s = C.c_uint64()
    lib().orc_tier_of(cap, cap_h, total, L, C.byref(t), C.byref(s))
    return int(t.value), int(s.value)

