"""The allocation-free priority update, through the C ABI.

edp_update_priorities_td_static serves callers that cannot allocate device
memory while they update priorities (for instance while a CUDA graph is being
captured, or under a runtime that hands out all device memory at start-up):
it keeps its per-pair scratch in a fixed per-device array instead of
allocating it.  Its results must equal those of the allocating
edp_update_priorities_td on the same arguments -- here compared on the whole
priority tree (leaves, every internal sum, the deferred and the running
maximum priority), bit for bit, after two calls in a row, and after two
calls queued back to back on one stream; and against the oracle.  This
file is collected last so that a failure here leaves every other test
already run.
"""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, check_tree, cuda, fx, tree_levels

pytestmark = pytest.mark.gpu

ALPHA, EPS = 0.6, 1e-6


def _twin_rings(orc, cap, n):
    frames, action, reward, done = fx.dqn_transitions(21, n)
    q = orc.priorities_from_td(fx.td_errors(21, n), ALPHA, EPS)
    rings = []
    for _ in range(2):
        m = MirroredDqn(cap, prioritized=True)
        m.ingest(orc, frames, action, reward, done, q=q)
        rings.append(m)
    return rings


def test_static_update_matches_allocating_update(edp_lib, orc):
    edp = edp_lib
    cap, n_ingest = 3000, 2500
    a, b = _twin_rings(orc, cap, n_ingest)
    rng = np.random.default_rng(22)
    for call in range(2):  # two calls in a row share the fixed array
        n = 700 + 300 * call
        idx = rng.integers(0, n_ingest, size=n).astype(np.int64)
        idx[::5] = idx[1]  # duplicates: the last pair wins
        idx[3] = n_ingest - 1  # the newest transition: deferred priority
        td = fx.td_errors(100 + call, n)
        td[:3] = [0.0, -4.0, 30.0]
        d_idx, d_td = cuda(idx), cuda(td)
        edp.edp_update_priorities_td(a.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
        edp.edp_update_priorities_td_static(b.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
        edp.edp_sync(a.ring.ctx)
        edp.edp_sync(b.ring.ctx)
        la, lva, pa, ma = tree_levels(a.ring)
        lb, lvb, pb, mb = tree_levels(b.ring)
        assert np.array_equal(la, lb), call
        for d, (x, y) in enumerate(zip(lva, lvb)):
            assert np.array_equal(x, y), (call, d)
        assert (pa, ma) == (pb, mb)
        # and the update did happen: the leaves of the updated slots moved
        assert not np.array_equal(la[:cap], b.st.leaves)
    # then a pair of calls queued back to back on one stream, with nothing
    # between them: stream order alone keeps them apart
    pairs = []
    for call in range(2):
        n = 4000
        idx = rng.integers(0, n_ingest, size=n).astype(np.int64)
        idx[: n // 2] = rng.integers(0, 300, size=n // 2)  # slots both calls hit
        pairs.append((cuda(idx), cuda(fx.td_errors(200 + call, n)), n))
    torch.cuda.synchronize()
    for d_idx, d_td, n in pairs:
        edp.edp_update_priorities_td(a.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
    for d_idx, d_td, n in pairs:
        edp.edp_update_priorities_td_static(b.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
    edp.edp_sync(a.ring.ctx)
    edp.edp_sync(b.ring.ctx)
    la, lva, pa, ma = tree_levels(a.ring)
    lb, lvb, pb, mb = tree_levels(b.ring)
    assert np.array_equal(la, lb)
    for d, (x, y) in enumerate(zip(lva, lvb)):
        assert np.array_equal(x, y), d
    assert (pa, ma) == (pb, mb)


def test_static_updates_back_to_back_match_oracle(edp_lib, orc):
    """Two calls of the allocation-free update queued straight after each
    other on one stream (no synchronisation, overlapping slots), then the
    whole tree bit for bit against the oracle applying both batches in
    order, with the priorities the device's rule gives for the same TD
    errors."""
    edp = edp_lib
    cap, n_ingest = 3000, 2500
    (m, _) = _twin_rings(orc, cap, n_ingest)
    rng = np.random.default_rng(23)
    calls = []
    for call in range(2):
        n = 5000
        idx = rng.integers(0, n_ingest, size=n).astype(np.int64)
        idx[: n // 2] = rng.integers(0, 400, size=n // 2)
        idx[9] = n_ingest - 1  # the newest transition: deferred priority
        d_td = cuda(fx.td_errors(300 + call, n))
        qd = torch.zeros(n, dtype=torch.int32, device="cuda")
        edp.edp_priorities_from_td(m.ring.ctx, d_td, n, ALPHA, EPS, qd)
        edp.edp_sync(m.ring.ctx)
        calls.append((cuda(idx), d_td, n, idx, qd.cpu().numpy().view(np.uint32)))
    torch.cuda.synchronize()
    for d_idx, d_td, n, _, _ in calls:
        edp.edp_update_priorities_td_static(m.ring.ctx, d_idx, d_td, n, ALPHA, EPS)
    edp.edp_sync(m.ring.ctx)
    for _, _, _, idx, q in calls:
        orc.update_leaves(m.st, m.total, idx, q)
    check_tree(orc, m.ring, m.st)


def test_static_update_rejects_sizes_above_its_maximum(edp_lib, orc):
    edp = edp_lib
    a, _ = _twin_rings(orc, 64, 40)
    n = 16385
    idx = torch.zeros(n, dtype=torch.int64, device="cuda")
    td = torch.ones(n, dtype=torch.float32, device="cuda")
    with pytest.raises(edp.EdpError) as e:
        edp.edp_update_priorities_td_static(a.ring.ctx, idx, td, n, ALPHA, EPS)
    assert e.value.status == edp.EDP_ERR_INVALID
    assert "16384" in str(e.value)
