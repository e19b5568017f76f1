"""The staged path of the frame-stack delivery, under concurrency.

A batch that fills the GPU (here 1,024 stacks, 5,120 frame pieces) is
delivered by the staged kernel: pieces are dealt to the CTAs round robin,
so a launch shares no state with any other and leaves none behind.  Here it
is delivered many times: from two streams at once, 40 times in a row inside
a CUDA graph, and 40 deliveries that may all run at once -- released
together on eight streams, eagerly and from a graph replayed twice.  Every
delivery must equal the first bit for bit, and the first must equal the
oracle on a strided sample of rows.
"""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, bits, dqn_outputs, fx, to_np

pytestmark = pytest.mark.gpu

B, CAP, N_INGEST = 1024, 3000, 2900


def test_concurrent_and_repeated_staged_deliveries(edp_lib, orc):
    edp = edp_lib
    frames, action, reward, done = fx.dqn_transitions(40, N_INGEST, done_p=0.05)
    m = MirroredDqn(CAP)
    m.ingest(orc, frames, action, reward, done)
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 41, 0, idx)
    outs = [dqn_outputs(B, m.K, m.F) for _ in range(4)]
    batches = [edp.make_batch(*o) for o in outs]
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    torch.cuda.synchronize()
    # two concurrent launches per stream pair, twice
    start = torch.cuda.Event()
    start.record()
    for i, b in enumerate(batches):
        st = streams[i % 2]
        st.wait_event(start)
        edp.edp_deliver(m.ring.ctx, idx, B, b, stream=st)
    torch.cuda.synchronize()
    edp.edp_sync(m.ring.ctx)
    ref = [bits(t) if t.is_floating_point() else to_np(t) for t in outs[0]]
    for o in outs[1:]:
        for x, y in zip(ref, o):
            assert np.array_equal(x, bits(y) if y.is_floating_point() else to_np(y))
    # the first delivery against the oracle on every 7th row
    sel = np.arange(0, B, 7)
    ref_idx = to_np(idx)
    r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
        m.frames, m.done, m.action, m.reward, m.cap, m.total, m.K, ref_idx[sel])
    assert np.array_equal(ref[0][sel].reshape(r_obs.shape), r_obs.view(np.uint32))
    assert np.array_equal(ref[1][sel].reshape(r_nxt.shape), r_nxt.view(np.uint32))
    assert np.array_equal(ref[2][sel], r_act)
    assert np.array_equal(ref[3][sel], r_rew.view(np.uint32))
    assert np.array_equal(ref[4][sel], r_dn)
    # 40 launches in one graph,
    # alternating between two output sets; the last two must equal ref
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        for i in range(40):
            edp.edp_deliver(m.ring.ctx, idx, B, batches[2 + i % 2])
    for o in outs[2:]:
        for t in o:
            t.fill_(7)
    g.replay()
    torch.cuda.synchronize()
    edp.edp_sync(m.ring.ctx)
    for o in outs[2:]:
        for x, y in zip(ref, o):
            assert np.array_equal(x, bits(y) if y.is_floating_point() else to_np(y))


@pytest.mark.parametrize("B", [37, 1024])
def test_outputs_16_byte_aligned_only(edp_lib, orc, B):
    """Outputs 16 bytes past a 32-byte boundary (the alignment the ABI
    requires, and no more) give the same batches as aligned ones, on the
    one-chunk-per-CTA and the staged paths."""
    edp = edp_lib
    frames, action, reward, done = fx.dqn_transitions(42, N_INGEST, done_p=0.05)
    m = MirroredDqn(CAP)
    m.ingest(orc, frames, action, reward, done)
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 43, 0, idx)
    n = B * 4 * m.F
    aligned = dqn_outputs(B, m.K, m.F)
    # each output 16 bytes past a fresh (256-byte aligned) allocation
    obs = torch.full((n + 4,), float("nan"), device="cuda")[4:].view(B, 4, m.F)
    nxt = torch.full((n + 4,), float("nan"), device="cuda")[4:].view(B, 4, m.F)
    assert obs.data_ptr() % 32 == 16 and nxt.data_ptr() % 32 == 16
    odd = (obs, nxt) + tuple(torch.empty_like(t) for t in aligned[2:])
    edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(*aligned))
    edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(*odd))
    edp.edp_sync(m.ring.ctx)
    for x, y in zip(aligned, odd):
        assert np.array_equal(bits(x) if x.is_floating_point() else to_np(x),
                              bits(y) if y.is_floating_point() else to_np(y))


def test_forty_deliveries_in_flight_at_once(edp_lib, orc):
    """40 large deliveries with no order between them (8 streams, released
    by one event; then the same as 40 independent nodes of one graph,
    replayed twice with the outputs overwritten in between, so that a
    replay that skipped its work would show), each into its own outputs."""
    edp = edp_lib
    B, n_out, n_streams = 256, 40, 8
    frames, action, reward, done = fx.dqn_transitions(44, N_INGEST, done_p=0.05)
    m = MirroredDqn(CAP)
    m.ingest(orc, frames, action, reward, done)
    idx = torch.empty(B, dtype=torch.int64, device="cuda")
    edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_UNIFORM, B, 45, 0, idx)
    first = dqn_outputs(B, m.K, m.F)
    edp.edp_deliver(m.ring.ctx, idx, B, edp.make_batch(*first))
    edp.edp_sync(m.ring.ctx)
    ref = [bits(t) if t.is_floating_point() else to_np(t) for t in first]
    sel = np.arange(0, B, 5)
    r_obs, r_nxt, r_act, r_rew, r_dn = orc.deliver_dqn(
        m.frames, m.done, m.action, m.reward, m.cap, m.total, m.K, to_np(idx)[sel])
    assert np.array_equal(ref[0][sel].reshape(r_obs.shape), r_obs.view(np.uint32))
    assert np.array_equal(ref[1][sel].reshape(r_nxt.shape), r_nxt.view(np.uint32))
    assert np.array_equal(ref[2][sel], r_act)
    assert np.array_equal(ref[4][sel], r_dn)
    outs = [dqn_outputs(B, m.K, m.F) for _ in range(n_out)]
    batches = [edp.make_batch(*o) for o in outs]
    streams = [torch.cuda.Stream() for _ in range(n_streams)]

    def check(tag):
        for i, o in enumerate(outs):
            for j, (x, y) in enumerate(zip(ref, o)):
                got = bits(y) if y.is_floating_point() else to_np(y)
                assert np.array_equal(x, got), (tag, i, j)

    torch.cuda.synchronize()
    go = torch.cuda.Event()
    go.record()
    for i, b in enumerate(batches):
        st = streams[i % n_streams]
        st.wait_event(go)
        edp.edp_deliver(m.ring.ctx, idx, B, b, stream=st)
    torch.cuda.synchronize()
    edp.edp_sync(m.ring.ctx)
    check("eager")
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        fork = torch.cuda.current_stream()
        for i, b in enumerate(batches):
            st = streams[i % n_streams]
            st.wait_stream(fork)
            edp.edp_deliver(m.ring.ctx, idx, B, b, stream=st)
        for st in streams:
            fork.wait_stream(st)
    for rep in range(2):
        for o in outs:
            for t in o:
                t.fill_(7)
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        edp.edp_sync(m.ring.ctx)
        check("replay %d" % rep)
