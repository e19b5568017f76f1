"""Error behaviour of the C ABI on the GPU: synchronous argument and state
errors, and device-detected faults reported by edp_sync without trapping
(outputs zeroed, context still usable)."""
import numpy as np
import pytest
import torch

from gpu_util import MirroredDqn, cuda, dqn_outputs, fx, to_np

pytestmark = pytest.mark.gpu


def test_sync_errors_and_recovery(edp_lib, orc):
    edp = edp_lib
    m = MirroredDqn(100)
    ctx = m.ring.ctx
    idx = torch.zeros(4, dtype=torch.int64, device="cuda")
    with pytest.raises(edp.EdpError) as e:  # empty ring
        edp.edp_sample(ctx, edp.EDP_SAMPLE_UNIFORM, 4, 0, 0, idx)
    assert e.value.status == edp.EDP_ERR_EMPTY
    frames, action, reward, done = fx.dqn_transitions(0, 50)
    m.ingest(orc, frames, action, reward, done)
    with pytest.raises(edp.EdpError) as e:  # no tree
        edp.edp_sample(ctx, edp.EDP_SAMPLE_PRIORITIZED, 4, 0, 0, idx)
    assert e.value.status == edp.EDP_ERR_STATE
    with pytest.raises(edp.EdpError) as e:  # batch 0
        edp.edp_sample(ctx, edp.EDP_SAMPLE_UNIFORM, 0, 0, 0, idx)
    assert e.value.status == edp.EDP_ERR_INVALID
    host_idx = torch.zeros(4, dtype=torch.int64)  # pageable host memory
    with pytest.raises(edp.EdpError) as e:
        edp.edp_sample(ctx, edp.EDP_SAMPLE_UNIFORM, 4, 0, 0, host_idx)
    assert e.value.status == edp.EDP_ERR_INVALID
    with pytest.raises(edp.EdpError) as e:  # n > capacity
        edp.edp_ingest(ctx, cuda(np.zeros((101, 7056), np.uint8)), 101)
    assert e.value.status == edp.EDP_ERR_INVALID
    # out-of-range and not-yet-sampleable slots: zeros + a flag at sync
    bad = cuda(np.array([3, 49, 120, -2], np.int64))  # 49 is the newest
    obs, nxt, act, rew, dn = dqn_outputs(4, 4, 7056)
    edp.edp_deliver(ctx, bad, 4, edp.make_batch(obs, nxt, act, rew, dn))
    status, msg = edp.edp_sync_status(ctx)
    assert status == edp.EDP_ERR_INVALID, msg
    o = to_np(obs)
    assert np.all(o[1:] == 0) and np.isfinite(o[0]).all() and o[0].any()
    assert to_np(act)[1:].tolist() == [0, 0, 0]
    # the flag is cleared and the context keeps working
    edp.edp_sample(ctx, edp.EDP_SAMPLE_UNIFORM, 4, 0, 0, idx)
    edp.edp_sync(ctx)


def test_create_rejects_bad_configs(edp_lib):
    edp = edp_lib
    cfg = edp.make_config(10, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                          frame_stack=4, next_obs=True)
    with pytest.raises(edp.EdpError):  # done field missing
        edp.Ring(cfg, done=False)
    cfg2 = edp.make_config(10, (3, 10, 10), edp.EDP_XFORM_CHW_NORM_BF16)
    with pytest.raises(edp.EdpError):  # 300 bytes, not a multiple of 16
        edp.Ring(cfg2)
    cfg3 = edp.make_config(10, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                           hbm_capacity=5)
    with pytest.raises(edp.EdpError):  # two tiers only for CHW_NORM_BF16
        edp.Ring(cfg3)


def test_failing_allocator(edp_lib, orc):
    """Fault injection on the host through the allocator callback.  A
    creation whose allocation fails returns EDP_ERR_OOM and holds nothing.
    A call whose scratch allocation fails returns EDP_ERR_OOM and leaves the
    context usable: the same call succeeds once memory is granted."""
    edp = edp_lib
    grant = {"n": 0}
    live = {}

    def _alloc(user, nbytes):
        if grant["n"] <= 0:
            return None
        grant["n"] -= 1
        t = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
        live[t.data_ptr()] = t
        return t.data_ptr()

    def _free(user, p):
        live.pop(p, None)

    alloc, free = edp.ALLOC_FN(_alloc), edp.FREE_FN(_free)  # kept alive here
    cfg = edp.make_config(64, (3, 16, 16), edp.EDP_XFORM_HWC_CHW_BF16)
    cfg.alloc, cfg.free = alloc, free
    with pytest.raises(edp.EdpError) as e:
        edp.Ring(cfg, action=False, reward=False, done=False)
    assert e.value.status == edp.EDP_ERR_OOM
    assert not live
    grant["n"] = 1  # the control block, and nothing more
    ring = edp.Ring(cfg, action=False, reward=False, done=False)
    assert len(live) == 1
    obs = torch.randint(0, 256, (64, 768), dtype=torch.uint8, device="cuda")
    edp.edp_ingest(ring.ctx, obs, 64)
    idx = torch.full((64,), -1, dtype=torch.int64, device="cuda")
    with pytest.raises(edp.EdpError) as e:  # the shuffle's scratch
        edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, 64, 5, 0, idx)
    assert e.value.status == edp.EDP_ERR_OOM
    grant["n"] = 4
    edp.edp_sample(ring.ctx, edp.EDP_SAMPLE_PERMUTE, 64, 5, 0, idx)
    edp.edp_sync(ring.ctx)
    assert np.array_equal(to_np(idx), orc.permutation(64, 5, 0))
    ring.close()
    assert not live  # everything libedp took went back through free


def test_scratch_growth_refused_during_capture(edp_lib, orc):
    """A call whose scratch would have to grow while its stream is being
    captured returns EDP_ERR_STATE and enqueues nothing (the capture stays
    usable); made once outside the capture, the same call then captures and
    replays to the oracle's result."""
    edp = edp_lib
    cfg = edp.make_config(64, (3, 16, 16), edp.EDP_XFORM_HWC_CHW_BF16)
    ring = edp.Ring(cfg, action=False, reward=False, done=False)
    T, E = 8, 16
    r = torch.randn(T, E, device="cuda")
    v = torch.randn(T + 1, E, device="cuda")
    d = torch.zeros(T, E, dtype=torch.uint8, device="cuda")
    adv = torch.zeros(T, E, device="cuda")
    ret = torch.zeros(T, E, device="cuda")
    nrm = torch.zeros(T, E, device="cuda")
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        with pytest.raises(edp.EdpError) as e:
            edp.edp_gae(ring.ctx, r, v, d, T, E, 0.99, 0.95, adv, ret, nrm)
    assert e.value.status == edp.EDP_ERR_STATE
    assert "captur" in str(e.value)
    edp.edp_gae(ring.ctx, r, v, d, T, E, 0.99, 0.95, adv, ret, nrm)  # grows here
    edp.edp_sync(ring.ctx)
    nrm.zero_()
    g2 = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g2, capture_error_mode="thread_local"):
        edp.edp_gae(ring.ctx, r, v, d, T, E, 0.99, 0.95, adv, ret, nrm)
    g2.replay()
    torch.cuda.synchronize()
    edp.edp_sync(ring.ctx)
    A, _ = orc.gae(to_np(r), to_np(v), to_np(d), 0.99, 0.95)
    N, _, _ = orc.normalize(A)
    assert np.abs(to_np(nrm) - N).max() <= 1e-5
    ring.close()


def test_calls_keep_the_callers_current_device(edp_lib, orc):
    """Every call on a context of device 0 leaves the calling thread's
    current device as it found it: device 0 here, and, where a second GPU
    exists, the other device made current before the calls."""
    edp = edp_lib
    homes = [0] + ([1] if torch.cuda.device_count() > 1 else [])
    m = MirroredDqn(100, prioritized=True)
    frames, action, reward, done = fx.dqn_transitions(3, 60)
    m.ingest(orc, frames, action, reward, done)
    idx = torch.zeros(8, dtype=torch.int64, device="cuda:0")
    q = torch.zeros(8, dtype=torch.int32, device="cuda:0")
    td = torch.ones(8, dtype=torch.float32, device="cuda:0")
    obs, nxt, act, rew, dn = dqn_outputs(8, 4, 7056)
    s0 = torch.cuda.Stream(device=0)
    for home in homes:
        torch.cuda.set_device(home)
        calls = [
            lambda: edp.edp_sample(m.ring.ctx, edp.EDP_SAMPLE_PRIORITIZED, 8, 1, 0, idx, q,
                                   stream=s0),
            lambda: edp.edp_deliver(m.ring.ctx, idx, 8, edp.make_batch(obs, nxt, act, rew, dn),
                                    stream=s0),
            lambda: edp.edp_update_priorities_td(m.ring.ctx, idx, td, 8, 0.6, 1e-6, stream=s0),
            lambda: edp.edp_update_priorities_td_static(m.ring.ctx, idx, td, 8, 0.6, 1e-6,
                                                        stream=s0),
            lambda: edp.edp_sync(m.ring.ctx, stream=s0),
        ]
        for call in calls:
            call()
            assert torch.cuda.current_device() == home
    torch.cuda.set_device(0)
