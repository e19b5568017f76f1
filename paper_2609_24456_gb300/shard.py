"""A buffer sharded across the GPUs of a node (the shared-GPU placement of
Sec. 5.1: each GPU holds a share of the ring's slots and every learner
samples the whole buffer, most of it from other GPUs).

Every step of the data path runs in libedp's kernels (include/edp.h,
"Sharded buffer"); this module sequences them and performs the exchanges
with torch.distributed collectives -- the one exchange a round needs:

- ``ShardedPer``: prioritized replay.  G ranks each own one shard (an edp
  context) and one learner, which receives strata [rank B_l, (rank+1) B_l)
  of every global batch of B = G B_l.  A round: shard totals all-gathered;
  each learner routes its stratified targets to the owning shards (counts,
  then targets, all-to-all); owners descend their trees and deliver the rows,
  which return with the reverse all-to-all in stratum order; the minimum
  priority of the global batch is reduced over ranks for the importance
  weights.  Priority updates go back to the owners in the same grouping.
  The result equals one buffer holding all shards' leaves in shard-major
  order.
- ``sharded_gae``: an on-policy rollout whose environments are split over
  the ranks: each rank's GAE and (n, sum A, sum A^2), one fp64 all-reduce,
  then the global normalisation.

``ShardComm`` runs the collectives on device tensors with a device
transport (NCCL); over gloo (the CPU transport of the multi-process tests)
it stages them through host memory.
"""
from . import edp


class ShardComm:
    """Collectives of the sharded path over a torch.distributed group."""

    def __init__(self, group=None):
        import torch.distributed as dist
        self.dist = dist
        self.group = group
        self.rank = dist.get_rank(group)
        self.world = dist.get_world_size(group)
        self.host = dist.get_backend(group) == "gloo"

    def _out(self, t):
        return t.cpu() if self.host and t.is_cuda else t

    def _back(self, src, res, out=None):
        if out is not None:
            out.copy_(res)
            return out
        return res.to(src.device) if res.device != src.device else res

    def all_gather(self, t, out=None):
        """[world * n] from every rank's [n] (rank order)."""
        import torch
        src = self._out(t.contiguous())
        if out is not None and not self.host:
            self.dist.all_gather_into_tensor(out, src, group=self.group)
            return out
        res = torch.empty(self.world * src.numel(), dtype=src.dtype, device=src.device)
        self.dist.all_gather_into_tensor(res, src, group=self.group)
        return self._back(t, res, out)

    def all_to_all(self, t, send_counts, recv_counts, out=None):
        """Rows [sum send_counts, ...] out, rows [sum recv_counts, ...] in:
        send_counts[s] consecutive rows go to rank s; the rows from rank s
        arrive in rank order."""
        import torch
        src = self._out(t.contiguous())
        n = sum(recv_counts)
        if out is not None and not self.host:
            res = out[:n]  # received in place (a leading slice is contiguous)
        else:
            res = torch.empty((n,) + tuple(src.shape[1:]), dtype=src.dtype, device=src.device)
        self.dist.all_to_all_single(res, src, output_split_sizes=list(recv_counts),
                                    input_split_sizes=list(send_counts), group=self.group)
        if out is not None:
            if res.data_ptr() != out.data_ptr() or res.device != out.device:
                out[:n].copy_(res)
            return out[:n]
        return self._back(t, res)

    def all_reduce(self, t, op):
        """In place: "sum" or "min" over the ranks."""
        ops = {"sum": self.dist.ReduceOp.SUM, "min": self.dist.ReduceOp.MIN}
        src = self._out(t)
        self.dist.all_reduce(src, op=ops[op], group=self.group)
        if src is not t:
            t.copy_(src)
        return t


class ShardedPer:
    """This rank's shard of a prioritized frame-stack replay buffer sharded
    over ``comm``'s ranks, and its learner's share of each global batch.

    ``ring`` is this rank's ``edp.Ring`` (a prioritized STACK_F32 context
    with next_obs); every rank's ring has the same layout.  A global batch
    holds ``batch_per_rank`` samples per rank.  ``sample_deliver`` returns
    this learner's rows in stratum order; ``update`` sends the learner's
    TD errors (or priorities) for those rows back to their owners."""

    def __init__(self, ring, comm, batch_per_rank, beta=0.4, alpha=0.6, eps=1e-6,
                 device=None):
        import torch
        self.ring, self.comm = ring, comm
        self.ctx = ring.ctx
        info = edp.edp_get_info(self.ctx)
        cfg = ring.cfg
        self.K = cfg.frame_stack
        self.F = cfg.obs_h * cfg.obs_w * cfg.obs_c
        self.G, self.rank = comm.world, comm.rank
        self.Bl = batch_per_rank
        self.B = self.G * batch_per_rank
        self.cap = info.capacity
        self.beta, self.alpha, self.eps = beta, alpha, eps
        dev = device or torch.device("cuda", cfg.device)
        self.device = dev
        i64 = dict(dtype=torch.int64, device=dev)
        B, Bl, K, F = self.B, self.Bl, self.K, self.F
        self.total = torch.zeros(1, **i64)
        self.totals = torch.zeros(self.G, **i64)
        self.local_t = torch.zeros(Bl, **i64)
        self.counts = torch.zeros(self.G, **i64)
        self.qmin = torch.zeros(1, **i64)
        # owner side: targets routed here by every learner (at most B)
        self.t_recv = torch.zeros(B, **i64)
        self.idx_recv = torch.zeros(B, **i64)
        self.q_recv = torch.zeros(B, dtype=torch.int32, device=dev)
        self.own = {"obs": torch.empty((B, K, F), device=dev),
                    "nxt": torch.empty((B, K, F), device=dev),
                    "act": torch.empty(B, dtype=torch.int32, device=dev),
                    "rew": torch.empty(B, device=dev),
                    "done": torch.empty(B, dtype=torch.uint8, device=dev)}
        # learner side
        self.out = {"obs": torch.empty((Bl, K, F), device=dev),
                    "nxt": torch.empty((Bl, K, F), device=dev),
                    "act": torch.empty(Bl, dtype=torch.int32, device=dev),
                    "rew": torch.empty(Bl, device=dev),
                    "done": torch.empty(Bl, dtype=torch.uint8, device=dev),
                    "idx": torch.empty(Bl, **i64),
                    "q": torch.empty(Bl, dtype=torch.int32, device=dev),
                    "isw": torch.empty(Bl, device=dev)}
        self.td_recv = torch.zeros(B, device=dev)
        self.q_upd = torch.zeros(B, dtype=torch.int32, device=dev)
        self.send_counts = self.recv_counts = None
        self.owner = None

    def sample_deliver(self, seed, round_):
        """One round of sampling and delivery; returns this learner's batch
        (dict of device tensors: obs, nxt, act, rew, done, idx = the slot in
        its owner's ring, q, isw) and ``owner`` (the owning rank per row)."""
        import torch
        ctx, comm = self.ctx, self.comm
        edp.edp_tree_total(ctx, self.total)
        comm.all_gather(self.total, out=self.totals)
        edp.edp_route_prioritized(ctx, self.totals, self.G, self.B, self.rank * self.Bl,
                                  self.Bl, seed, round_, self.local_t, self.counts)
        send = [int(c) for c in self.counts.tolist()]  # waits for the routing
        if sum(send) != self.Bl:
            edp.edp_sync(ctx)  # raises: the device flagged an empty distribution
            raise edp.EdpError(edp.EDP_ERR_EMPTY, "sharded sampling routed no stratum")
        counts_in = comm.all_to_all(self.counts, [1] * self.G, [1] * self.G)
        recv = [int(c) for c in counts_in.tolist()]
        n = sum(recv)
        comm.all_to_all(self.local_t, send, recv, out=self.t_recv)
        o = self.own
        if n:
            edp.edp_sample_targets(ctx, self.t_recv, n, self.idx_recv, self.q_recv)
            batch = edp.make_batch(o["obs"][:n], o["nxt"][:n], o["act"][:n], o["rew"][:n],
                                   o["done"][:n])
            edp.edp_deliver(ctx, self.idx_recv, n, batch)
        # rows back to their learners, in stratum order
        lo = self.out
        for key in ("obs", "nxt", "act", "rew", "done"):
            comm.all_to_all(o[key][:n], recv, send, out=lo[key])
        comm.all_to_all(self.idx_recv[:n], recv, send, out=lo["idx"])
        comm.all_to_all(self.q_recv[:n], recv, send, out=lo["q"])
        # importance weights against the minimum over the global batch
        edp.edp_batch_qmin(ctx, lo["q"], self.Bl, self.qmin)
        comm.all_reduce(self.qmin, "min")
        edp.edp_is_weights(ctx, lo["q"], self.Bl, self.qmin, self.beta, lo["isw"])
        self.send_counts, self.recv_counts, self.n_recv = send, recv, n
        self.owner = torch.repeat_interleave(torch.arange(self.G), torch.tensor(send))
        return lo, self.owner

    def update(self, td=None, q=None):
        """Priority update of the last round's rows from this learner's TD
        errors (device float [B_l]) or priorities (device uint32 [B_l], as
        int32), in batch order: they travel to the owners, which apply every
        learner's pairs in global batch order (the last occurrence of a slot
        wins) with edp_update_priorities_td / edp_update_priorities."""
        if (td is None) == (q is None):
            raise ValueError("ShardedPer.update: give exactly one of td and q")
        n = self.n_recv
        vals = td if td is not None else q
        buf = self.td_recv if td is not None else self.q_upd
        self.comm.all_to_all(vals, self.send_counts, self.recv_counts, out=buf)
        if not n:
            return
        if td is not None:
            edp.edp_update_priorities_td(self.ctx, self.idx_recv, buf, n, self.alpha,
                                         self.eps)
        else:
            edp.edp_update_priorities(self.ctx, self.idx_recv, buf, n)


def sharded_gae(ctx, comm, r, v, d, T, E, gamma, lam, adv, ret, adv_norm, stats):
    """GAE over this rank's E environments with the advantage normalisation
    over every rank's T x E values: edp_gae_stats, a sum of (n, sum A,
    sum A^2) over the ranks, edp_gae_normalize.  ``stats`` is a device fp64
    [3] buffer."""
    edp.edp_gae_stats(ctx, r, v, d, T, E, gamma, lam, adv, stats, ret=ret)
    comm.all_reduce(stats, "sum")
    edp.edp_gae_normalize(ctx, adv, T * E, stats, adv_norm)
