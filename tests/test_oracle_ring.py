"""Pins of the oracle's ring (FIFO eviction) and frame-stack delivery.

The ring is checked against a brute-force list model; frame stacks against
expectations enumerated by hand for episodes ending at offsets 0..3 and
across the wrap boundary (Mnih et al. frame stacking with zero padding at
episode starts).
"""
import numpy as np
import pytest


def test_ring_against_list_model(orc):
    rng = np.random.default_rng(11)
    for cap in range(1, 18):
        ring = np.zeros((cap, 3), np.uint8)
        act = np.zeros(cap, np.int32)  # a multi-byte field beside it
        model, amodel = [], []  # logical history of records
        total = 0
        for _ in range(12):
            n = int(rng.integers(0, cap + 1))
            src = rng.integers(0, 256, size=(n, 3), dtype=np.uint8)
            a = rng.integers(-2**31, 2**31, size=n, dtype=np.int32)
            orc.ring_write(ring, cap, total, src)
            orc.ring_write(act, cap, total, a)
            model.extend(src.tolist())
            amodel.extend(a.tolist())
            total += n
            size = orc.ring_size(cap, total)
            assert size == min(total, cap)
            kept = model[len(model) - size:]
            akept = amodel[len(amodel) - size:]
            for k in range(size):
                s = orc.ring_slot(cap, total, k)
                assert ring[s].tolist() == kept[k]
                assert int(act[s]) == akept[k]
                assert orc.ring_offset(cap, total, s) == k
                # logical id total-size+k lives in slot id mod cap
                assert s == (total - size + k) % cap


def _frames(cap):
    # frame of slot s is filled with byte s+1 so stacks are readable by value
    return np.repeat(np.arange(1, cap + 1, dtype=np.uint8)[:, None], 16, axis=1)


def _ids(stack):
    """Map a delivered [K, F] stack back to frame ids (0 = zero frame)."""
    out = []
    for row in stack:
        assert np.all(row == row[0])
        out.append(int(round(float(row[0]) * 255)))
    return out


def _check(orc, done_slots, cap, total, slot, exp_obs, exp_next, K=4):
    frames = _frames(cap)
    done = np.zeros(cap, np.uint8)
    done[list(done_slots)] = 1
    obs, nxt = orc.dqn_stack(frames, done, cap, total, K, slot)
    assert _ids(obs) == exp_obs
    assert _ids(nxt) == exp_next


# (done slots, anchor slot, expected obs ids, expected next_obs ids); cap=10,
# total=10 (no wrap, oldest = slot 0); ids are slot+1.
CASES = [
    # no episode end nearby
    ((), 5, [3, 4, 5, 6], [4, 5, 6, 7]),
    # anchor itself ends the episode: next_obs starts a new one
    ((5,), 5, [3, 4, 5, 6], [0, 0, 0, 7]),
    # episode ended one step before the anchor
    ((4,), 5, [0, 0, 0, 6], [0, 0, 6, 7]),
    # two steps before
    ((3,), 5, [0, 0, 5, 6], [0, 5, 6, 7]),
    # three steps before
    ((2,), 5, [0, 4, 5, 6], [4, 5, 6, 7]),
    # four steps before: only next_obs window... both clear of it
    ((1,), 5, [3, 4, 5, 6], [4, 5, 6, 7]),
    # near the oldest transition: frames before it are zero
    ((), 1, [0, 0, 1, 2], [0, 1, 2, 3]),
    ((), 0, [0, 0, 0, 1], [0, 0, 1, 2]),
    ((0,), 0, [0, 0, 0, 1], [0, 0, 0, 2]),
    # two episode ends inside the window
    ((2, 4), 5, [0, 0, 0, 6], [0, 0, 6, 7]),
]


@pytest.mark.parametrize("done_slots,slot,exp_obs,exp_next", CASES)
def test_frame_stack_hand_cases(orc, done_slots, slot, exp_obs, exp_next):
    _check(orc, done_slots, 10, 10, slot, exp_obs, exp_next)


def test_frame_stack_across_wrap(orc):
    # cap 6, total 9: ids 3..8 live in slots 3,4,5,0,1,2; oldest slot 3.
    cap, total = 6, 9
    # anchor offset 1 = id 4 (slot 4): offsets -2, -1 do not exist
    _check(orc, (), cap, total, 4, [0, 0, 4, 5], [0, 4, 5, 6])
    # anchor offset 3 = id 6 (slot 0); frames cross the physical wrap
    _check(orc, (), cap, total, 0, [4, 5, 6, 1], [5, 6, 1, 2])
    # episode end at id 5 (slot 5)
    _check(orc, (5,), cap, total, 0, [0, 0, 0, 1], [0, 0, 1, 2])


def test_frame_stack_k1_and_k2(orc):
    _check(orc, (5,), 10, 10, 5, [6], [7], K=1)
    _check(orc, (4,), 10, 10, 5, [0, 6], [6, 7], K=2)


def test_deliver_dqn_collates(orc):
    cap = 10
    frames = _frames(cap)
    done = np.zeros(cap, np.uint8)
    done[3] = 1
    action = np.arange(cap, dtype=np.int32) * 3
    reward = np.arange(cap, dtype=np.float32) - 4.5
    idx = np.array([3, 7, 3], np.int64)
    obs, nxt, act, rew, dn = orc.deliver_dqn(frames, done, action, reward, cap,
                                             cap, 4, idx)
    assert obs.shape == (3, 4, 16)
    assert act.tolist() == [9, 21, 9]
    assert rew.tolist() == [-1.5, 2.5, -1.5]
    assert dn.tolist() == [1, 0, 1]
    assert _ids(nxt[0]) == [0, 0, 0, 5]
