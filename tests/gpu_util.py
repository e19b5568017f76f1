"""Helpers shared by the GPU parity tests: device-pointer views and rings
mirrored in the oracle.  Inputs come from the fixture generators; expected
values come only from the oracle."""
import numpy as np
import torch

from paper_2609_24456_gb300 import edp
from paper_2609_24456_gb300 import fixtures as fx

# unsigned 32/64-bit device data is viewed through the signed torch dtypes
# (torch's unsigned support is partial) and reinterpreted on the host
_TYPESTR = {np.uint32: "<i4", np.uint64: "<i8", np.int64: "<i8",
            np.uint8: "|u1", np.float32: "<f4", np.int32: "<i4"}
_SIGNED = {np.dtype(np.uint32): np.int32, np.dtype(np.uint64): np.int64,
           np.dtype(np.uint16): np.int16}


class _DevArray:
    def __init__(self, p, n, dtype):
        self.__cuda_array_interface__ = {
            "shape": (n,), "typestr": _TYPESTR[dtype], "data": (p, False),
            "version": 2}


def dev_view(p, n, dtype):
    """torch tensor aliasing n elements at device address p (no copy)."""
    return torch.as_tensor(_DevArray(p, n, dtype), device="cuda")


def to_np(t):
    return t.detach().cpu().numpy()


def bits(t):
    """Raw bit pattern of a float32 / bfloat16 tensor as a numpy array."""
    if t.dtype == torch.bfloat16:
        return to_np(t.view(torch.int16)).view(np.uint16)
    if t.dtype == torch.float32:
        return to_np(t.view(torch.int32)).view(np.uint32)
    return to_np(t)


def tree_levels(ring):
    """(leaves, [level 0, ..., level D-1]) of a prioritized ring, copied."""
    info = ring.info()
    D = info.tree_depth
    u32 = lambda p, n: to_np(dev_view(p, n, np.uint32)).view(np.uint32)
    leaves = u32(info.tree_leaves, 32 ** D)
    lv = [to_np(dev_view(info.tree_level[d], 32 ** d, np.uint64)).view(np.uint64)
          for d in range(D)]
    pending = int(u32(info.pending_q, 1)[0])
    qmax = int(u32(info.max_q, 1)[0])
    return leaves, lv, pending, qmax


def check_tree(orc, ring, st):
    """Device tree == oracle leaves; every node == oracle sum of its range."""
    leaves, lv, pending, qmax = tree_levels(ring)
    cap = st.cap
    assert np.array_equal(leaves[:cap], st.leaves)
    assert not leaves[cap:].any()
    D = len(lv)
    # node n of level d covers leaves [n 32^(D-d), (n+1) 32^(D-d))
    padded = np.zeros(32 ** D, np.uint64)
    padded[:cap] = st.leaves
    for d in range(D):
        span = 32 ** (D - d)
        ref = padded.reshape(-1, span).sum(axis=1, dtype=np.uint64)
        assert np.array_equal(lv[d], ref), "level %d" % d
    # the root against the oracle's own exact sum
    assert int(lv[0][0]) == orc.leaf_sum(st.leaves, 0, cap)
    assert pending == int(st.pending[0])
    assert qmax == int(st.qmax[0])


def cuda(x):
    x = np.ascontiguousarray(x)
    if x.dtype in _SIGNED:
        x = x.view(_SIGNED[x.dtype])
    return torch.from_numpy(x).cuda()


def u32(t):
    """numpy uint32 view of an int32 device tensor holding uint32 data."""
    return to_np(t).view(np.uint32)


class MirroredDqn:
    """A STACK_F32 ring on the GPU and the same ring in host arrays for the
    oracle; ingest feeds both from the same fixture inputs."""

    def __init__(self, cap, K=4, next_obs=True, prioritized=False, F=84 * 84):
        self.cap, self.K, self.F = cap, K, F
        cfg = edp.make_config(cap, (1, 84, F // 84), edp.EDP_XFORM_STACK_F32,
                              frame_stack=K, next_obs=next_obs,
                              prioritized=prioritized)
        self.ring = edp.Ring(cfg)
        self.frames = np.zeros((cap, F), np.uint8)
        self.action = np.zeros(cap, np.int32)
        self.reward = np.zeros(cap, np.float32)
        self.done = np.zeros(cap, np.uint8)
        self.total = 0
        self.st = None
        if prioritized:
            from oracle import PerState
            self.st = PerState(cap, next_obs)

    def ingest(self, orc, frames, action, reward, done, q=None):
        n = len(action)
        edp.edp_ingest(self.ring.ctx, cuda(frames), n, action=cuda(action),
                       reward=cuda(reward), done=cuda(done),
                       q=None if q is None else cuda(q))
        orc.ring_write(self.frames, self.cap, self.total, np.ascontiguousarray(frames))
        orc.ring_write(self.action, self.cap, self.total, action)
        orc.ring_write(self.reward, self.cap, self.total, reward)
        orc.ring_write(self.done, self.cap, self.total, done)
        if self.st is not None:
            if q is None:
                orc.ingest_leaves_default(self.st, self.total, n)
            else:
                orc.ingest_leaves(self.st, self.total, q)
        self.total += n


def dqn_outputs(B, K, F, with_next=True):
    dev = "cuda"
    obs = torch.full((B, K, F), float("nan"), dtype=torch.float32, device=dev)
    nxt = (torch.full((B, K, F), float("nan"), dtype=torch.float32, device=dev)
           if with_next else None)
    act = torch.full((B,), -7, dtype=torch.int32, device=dev)
    rew = torch.full((B,), float("nan"), dtype=torch.float32, device=dev)
    dn = torch.full((B,), 9, dtype=torch.uint8, device=dev)
    return obs, nxt, act, rew, dn


__all__ = ["dev_view", "to_np", "bits", "tree_levels", "check_tree", "cuda", "u32",
           "MirroredDqn", "dqn_outputs", "fx"]
