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
