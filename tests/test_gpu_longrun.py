"""Parity at the configured run lengths, through the round schedules the
benchmark times: bench.py's own workload classes and round functions, the
rounds captured into CUDA graphs (one per segment of up to 50 rounds) and
replayed, exactly as the benchmark replays its timed region.

- Prioritized replay, 1,000,000 84x84 frames, batch 512: 1,000 rounds of
  stratified sampling -> fused frame-stack delivery -> priority update from
  TD errors, in the overlapped schedule (each delivery on one of two side
  streams, four rotating output sets, the update and the next sampling on
  the main stream).  Every round: indices and priorities bit-exact and IS
  weights within 1 ulp against the oracle sampling its own leaves, which it
  updates with its own priorities from the same TD errors.  After round 0,
  every 50th round and the last: the whole tree bit-exact, and that round's
  whole batch (obs, next_obs, action, reward, done) bit-exact.
- Multimodal replay, 200,000 transitions of 3x224x224 + 512 tokens, batch
  1,024: 500 rounds of the fused sample+deliver schedule (calls alternating
  between two side streams).  Indices every round; the whole batch (bf16
  image, tokens, reward) on rounds 0, every 50th and the last.
- Two-tier ring, 1,600,000 transitions (newest 800,000 in HBM, oldest
  800,000 in page-locked host memory), 4,096 transitions ingested per round
  from page-locked staging, batch 1,024: 500 rounds of ingest -> sample ->
  deliver.  Indices every round; the whole batch and the tier and slot of
  retained ids (both ends of each tier and a random sample) on rounds 0,
  every 50th and the last.

Each round's indices (and for PER priorities and weights) are copied into
a log by the stream that consumed them, after the consuming kernel, so the
schedule's order of kernels is otherwise unchanged.
"""
import gc

import numpy as np
import pytest
import torch

import bench
from gpu_util import bits, check_tree, fx, to_np

pytestmark = pytest.mark.gpu

CHECK_EVERY = 50


def _segments(rounds, every=CHECK_EVERY):
    """Consecutive round ranges ending at the checked rounds: 0, every,
    2 every, ..., rounds - 1."""
    ends = [0] + list(range(every, rounds - 1, every)) + [rounds - 1]
    segs, lo = [], 0
    for e in ends:
        segs.append(range(lo, e + 1))
        lo = e + 1
    return segs


def _run(wl, fn, seg, graph):
    """Rounds seg of fn, eagerly or captured into a graph and replayed once."""
    if not graph:
        for r in seg:
            fn(r)
        wl.join()
        return
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        for r in seg:
            fn(r)
        wl.join()
    g.replay()
    torch.cuda.synchronize()
    del g


def _ulps(a, b):
    a = np.asarray(a, np.float32).view(np.int32).astype(np.int64)
    b = np.asarray(b, np.float32).view(np.int32).astype(np.int64)
    return int(np.abs(a - b).max())


class _LoggedPer(bench.PerReplay):
    """The benchmark's prioritized replay; each round's indices, priorities
    and IS weights are copied to a log on the delivery's side stream, after
    the delivery, before the output set can be reused."""

    def add_log(self, rounds, device):
        B = self.B
        self.log = {"idx": torch.empty((rounds, B), dtype=torch.int64, device=device),
                    "q": torch.empty((rounds, B), dtype=torch.int32, device=device),
                    "isw": torch.empty((rounds, B), dtype=torch.float32, device=device)}

    def round_overlap(self, r):
        self._r = r
        super().round_overlap(r)

    def _overlapped(self, k, sample, deliver, after=None):
        r, o = self._r, self.outs[k]

        def deliver_and_log(st):
            deliver(st)
            for key, t in self.log.items():
                t[r].copy_(o[key])

        super()._overlapped(k, sample, deliver_and_log, after)


def test_prioritized_replay_1000_rounds_overlapped(edp_lib, orc):
    edp = edp_lib
    device = torch.device("cuda", 0)
    rounds = 1000
    wl = _LoggedPer()
    wl.setup(device)
    try:
        wl.add_log(rounds, device)
        cap, B, K, F, seed = wl.cap, wl.B, wl.K, wl.F, wl.seed
        # the oracle's replay from the same fixture inputs
        _, action, reward, done = fx.dqn_transitions(seed, cap, with_frames=False)
        st = orc.PerState(cap, True)
        orc.ingest_leaves(st, 0, orc.priorities_from_td(fx.td_errors(seed, cap),
                                                        bench.ALPHA, bench.EPS))
        check_tree(orc, wl.ring, st)
        td_q = [orc.priorities_from_td(fx.td_errors(seed, B, r), bench.ALPHA, bench.EPS)
                for r in range(wl.td_rounds)]
        frames = np.zeros((cap, F), np.uint8)  # filled where a checked batch reads
        have = np.zeros(cap, bool)
        for i, seg in enumerate(_segments(rounds)):
            # round 0 eagerly: its update allocates the priority scratch
            _run(wl, wl.round_overlap, seg, graph=i > 0)
            torch.cuda.synchronize()
            edp.edp_sync(wl.ring.ctx)
            lg = {k: to_np(v[seg.start:seg.stop]) for k, v in wl.log.items()}
            for j, r in enumerate(seg):
                ref_idx, ref_q = orc.sample_prioritized_bisect(st.leaves, B, seed, r)
                assert np.array_equal(lg["idx"][j], ref_idx), r
                assert np.array_equal(lg["q"][j].view(np.uint32), ref_q), r
                assert _ulps(lg["isw"][j], orc.is_weights(ref_q, bench.BETA)) <= 1, r
                orc.update_leaves(st, cap, ref_idx, td_q[r % wl.td_rounds])
            check_tree(orc, wl.ring, st)
            # the whole batch of the segment's last round (ids == slots: the
            # ring was filled exactly once)
            r = seg[-1]
            o = wl.outs[r % wl.R]
            need = np.unique((ref_idx[:, None] + np.arange(-3, 2)[None, :]) % cap)
            new = need[~have[need]]
            if len(new):
                frames[new] = fx.content_bytes(seed, new, F)
                have[new] = True
            r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
                frames, done, action, reward, cap, cap, K, ref_idx)
            assert np.array_equal(bits(o["obs"]).reshape(r_obs.shape), r_obs.view(np.uint32)), r
            assert np.array_equal(bits(o["nxt"]).reshape(r_nxt.shape), r_nxt.view(np.uint32)), r
            assert np.array_equal(to_np(o["act"]), r_act), r
            assert np.array_equal(bits(o["rew"]), r_rew.view(np.uint32)), r
            assert np.array_equal(to_np(o["done"]), r_dn), r
    finally:
        wl.ring.close()
        del wl
        gc.collect()
        torch.cuda.empty_cache()


class _LoggedMm(bench.MmReplay):
    """The benchmark's multimodal (or two-tier) replay with each round's
    indices copied to a log by the stream that delivered the round."""

    def add_log(self, rounds, device):
        self.log_idx = torch.empty((rounds, self.B), dtype=torch.int64, device=device)

    def round_fused(self, r):
        super().round_fused(r)
        k = r % 2
        with torch.cuda.stream(self.sides[k]):
            self.log_idx[r].copy_(self.outs[k]["idx"])

    def round(self, r):
        super().round(r)
        self.log_idx[r].copy_(self.outs[r % 2]["idx"])


def _check_mm_batch(orc, o, seed, cid, rid, rew_all, r):
    """The whole delivered batch against the oracle's normalisation of the
    content of the sampled transitions (content id cid, reward id rid)."""
    C, H, W, L = bench.MmReplay.C, bench.MmReplay.H, bench.MmReplay.W, bench.MmReplay.L
    B = len(cid)
    r_obs, r_tok, r_rew = orc.deliver_mm(
        fx.content_bytes(seed, cid, C * H * W), fx.token_content(seed, cid, L),
        rew_all[rid], C, H * W, np.arange(B), bench.MEAN3, bench.STD3)
    assert np.array_equal(bits(o["obs"]).reshape(B, -1), r_obs), r
    assert np.array_equal(to_np(o["tok"]), r_tok), r
    assert np.array_equal(bits(o["rew"]), r_rew.view(np.uint32)), r


def test_multimodal_replay_500_rounds_fused(edp_lib, orc):
    edp = edp_lib
    device = torch.device("cuda", 0)
    rounds = 500
    wl = _LoggedMm()
    wl.setup(device)
    try:
        wl.add_log(rounds, device)
        cap, B, seed = wl.cap, wl.B, wl.seed
        for i, seg in enumerate(_segments(rounds)):
            _run(wl, wl.round_fused, seg, graph=i > 0)
            torch.cuda.synchronize()
            edp.edp_sync(wl.ring.ctx)
            lg = to_np(wl.log_idx[seg.start:seg.stop])
            for j, r in enumerate(seg):
                ref_idx = orc.sample_uniform(cap, cap, cap, B, seed, r)
                assert np.array_equal(lg[j], ref_idx), r
            r = seg[-1]
            # ids == slots (filled exactly once)
            _check_mm_batch(orc, wl.outs[r % 2], seed, ref_idx, ref_idx, wl.rew_all, r)
    finally:
        wl.ring.close()
        del wl
        gc.collect()
        torch.cuda.empty_cache()


def test_two_tier_500_rounds(edp_lib, orc):
    edp = edp_lib
    device = torch.device("cuda", 0)
    rounds = 500
    wl = _LoggedMm(capacity=1_600_000, hbm_frac=0.5, ingest=4096)
    wl.setup(device)
    try:
        wl.add_log(rounds, device)
        cap, cap_h, B, seed, n_in = wl.cap, wl.cap_h, wl.B, wl.seed, wl.ingest
        F = wl.F
        rng = np.random.default_rng(seed)

        # every round ingests the same staged rows: ids >= cap hold content
        # ids cap .. cap + n_in - 1 and rewards 0 .. n_in - 1, in turn
        def content_id(L):
            return np.where(L < cap, L, cap + (L - cap) % n_in)

        def reward_id(L):
            return np.where(L < cap, L, (L - cap) % n_in)

        for i, seg in enumerate(_segments(rounds)):
            _run(wl, wl.round, seg, graph=i > 0)
            torch.cuda.synchronize()
            edp.edp_sync(wl.ring.ctx)
            lg = to_np(wl.log_idx[seg.start:seg.stop])
            for j, r in enumerate(seg):
                total = cap + n_in * (r + 1)
                ref_idx = orc.sample_uniform(cap, total, cap, B, seed, r)
                assert np.array_equal(lg[j], ref_idx), r
            r = seg[-1]
            total = cap + n_in * (r + 1)
            assert wl.ring.info().total == total
            oldest = total % cap
            ids = total - cap + (ref_idx - oldest) % cap
            _check_mm_batch(orc, wl.outs[r % 2], seed, content_id(ids), reward_id(ids),
                            wl.rew_all, r)
            # placement of retained ids: both ends of each tier, and a sample
            probe = np.concatenate([[total - cap, total - cap_h - 1, total - cap_h, total - 1],
                                    rng.integers(total - cap, total, size=12)])
            for Lid in probe:
                tier, slot = orc.tier_of(cap, cap_h, total, int(Lid))
                assert tier == (0 if Lid >= total - cap_h else 1), (r, Lid)
                row = (wl.ring.host_obs[slot].numpy() if tier == 1
                       else wl.ring.obs[slot].cpu().numpy())
                want = fx.content_bytes(seed, [int(content_id(np.int64(Lid)))], F)[0]
                assert np.array_equal(row, want), (r, Lid)
    finally:
        wl.ring.close()
        for name in ("st_obs", "st_tok", "st_rew"):
            if hasattr(wl, name):
                delattr(wl, name)
        del wl
        gc.collect()
        torch.cuda.empty_cache()
        if hasattr(torch._C, "_host_emptyCache"):
            torch._C._host_emptyCache()  # the 122 GB of page-locked host tier
