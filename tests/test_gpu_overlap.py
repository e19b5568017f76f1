"""The overlapped round schedule gives the results of the serial one.

A round of prioritized replay is sample -> deliver -> priority update.  The
delivery depends only on the sampled indices, so it may run on a second
stream while the update and the next round's sampling run on the first (the
overlapped timing of Sec. 6.1); with two side streams consecutive deliveries
may also overlap each other.  With the dependencies kept -- delivery r
after sampling r, sampling r+1 after update r, and sampling r+R after
delivery r has read the R-th previous index set -- every sampled index, every
delivered batch and the final priority tree must equal, bit for bit, those of
the one-stream schedule, run eagerly and inside a CUDA graph.
"""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, dqn_outputs, fx, to_np, tree_levels

pytestmark = pytest.mark.gpu

ALPHA, EPS, BETA = 0.6, 1e-6, 0.4
CAP, N_INGEST, B, ROUNDS, R, F = 3000, 2500, 256, 12, 2, 84 * 16


class _Rounds:
    def __init__(self, edp, orc, frames, action, reward, done, q):
        self.edp = edp
        self.m = MirroredDqn(CAP, prioritized=True, F=F)
        self.m.ingest(orc, frames, action, reward, done, q=q)
        dev = "cuda"
        # R rotating index sets (the reuse the schedule must guard), one
        # output batch per round so that every round can be compared
        self.idx = [torch.zeros(B, dtype=torch.int64, device=dev) for _ in range(R)]
        self.q = [torch.zeros(B, dtype=torch.int32, device=dev) for _ in range(R)]
        self.out = []
        for _ in range(ROUNDS):
            obs, nxt, act, rew, dn = dqn_outputs(B, 4, F)
            isw = torch.zeros(B, dtype=torch.float32, device=dev)
            idx_copy = torch.zeros(B, dtype=torch.int64, device=dev)
            self.out.append((obs, nxt, act, rew, dn, isw, idx_copy))
        self.td = [torch.from_numpy(fx.td_errors(31, B, r)).cuda() for r in range(ROUNDS)]
        self.sides = [torch.cuda.Stream(), torch.cuda.Stream()]
        self.ready = [torch.cuda.Event() for _ in range(R)]
        self.consumed = [torch.cuda.Event() for _ in range(R)]

    def _sample(self, r):
        k = r % R
        self.edp.edp_sample(self.m.ring.ctx, self.edp.EDP_SAMPLE_PRIORITIZED, B,
                            77, r, self.idx[k], self.q[k])

    def _deliver(self, r, stream=None):
        k = r % R
        self._deliver_into(self.idx[k], self.q[k], self.out[r], stream)

    def _update(self, r):
        self.edp.edp_update_priorities_td(self.m.ring.ctx, self.idx[r % R], self.td[r],
                                          B, ALPHA, EPS)

    def warm(self):
        """One eager round, the same on every run: it makes the context's
        scratch allocations before any graph capture."""
        self.edp.edp_sample(self.m.ring.ctx, self.edp.EDP_SAMPLE_PRIORITIZED, B,
                            77, 1000, self.idx[0], self.q[0])
        self._deliver_into(self.idx[0], self.q[0], self.out[0])
        self.edp.edp_update_priorities_td(self.m.ring.ctx, self.idx[0], self.td[0],
                                          B, ALPHA, EPS)

    def _deliver_into(self, idx, q, out, stream=None):
        obs, nxt, act, rew, dn, isw, idx_copy = out
        self.edp.edp_deliver(self.m.ring.ctx, idx, B,
                             self.edp.make_batch(obs, nxt, act, rew, dn, q=q,
                                                 isw=isw, beta=BETA), stream=stream)
        idx_copy.copy_(idx)

    def serial(self):
        for r in range(ROUNDS):
            self._sample(r)
            self._deliver(r)
            self._update(r)

    def overlapped(self, nsides):
        main = torch.cuda.current_stream()
        for r in range(ROUNDS):
            k = r % R
            if r >= R:
                main.wait_event(self.consumed[k])
            self._sample(r)
            self.ready[k].record()
            side = self.sides[r % nsides]  # consecutive deliveries may overlap
            with torch.cuda.stream(side):
                side.wait_event(self.ready[k])
                self._deliver(r, stream=side)
                self.consumed[k].record()
            self._update(r)
        for side in self.sides[:nsides]:
            main.wait_stream(side)

    def results(self):
        self.edp.edp_sync(self.m.ring.ctx)
        torch.cuda.synchronize()
        per_round = [tuple(bits(t) if t.is_floating_point() else to_np(t) for t in o)
                     for o in self.out]
        leaves, lv, pending, qmax = tree_levels(self.m.ring)
        return per_round, (leaves, lv, pending, qmax)


@pytest.mark.parametrize("nsides", [1, 2])
def test_overlapped_rounds_equal_serial_rounds(edp_lib, orc, nsides):
    edp = edp_lib
    frames, action, reward, done = fx.dqn_transitions(30, N_INGEST, F)
    q = orc.priorities_from_td(fx.td_errors(30, N_INGEST), ALPHA, EPS)
    runs = [_Rounds(edp, orc, frames, action, reward, done, q) for _ in range(3)]
    for run in runs:
        run.warm()
    torch.cuda.synchronize()
    runs[0].serial()
    runs[1].overlapped(nsides)
    g = torch.cuda.CUDAGraph()
    torch.cuda.synchronize()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        runs[2].overlapped(nsides)
    g.replay()
    ref_rounds, ref_tree = runs[0].results()
    # the rounds did change the tree and sampled more than one index set
    assert len({r[-1].tobytes() for r in ref_rounds}) == ROUNDS
    for run in runs[1:]:
        rounds, tree = run.results()
        for r, (a, b) in enumerate(zip(ref_rounds, rounds)):
            for j, (x, y) in enumerate(zip(a, b)):
                assert np.array_equal(x, y), (r, j)
        assert np.array_equal(ref_tree[0], tree[0])
        for x, y in zip(ref_tree[1], tree[1]):
            assert np.array_equal(x, y)
        assert ref_tree[2:] == tree[2:]
