"""Randomised packed deliveries against the oracle: rollouts of 1 to 400
sequences whose lengths mix empty, short (under one 16-byte run) and long
(several 4,096-token bulk copies) ones, sources and outputs at every
4-byte offset from a 16-byte boundary, batches of 1 to 3,000 entries with
repeats and indices outside the rollout, with and without per-token
values, and an output capacity that sometimes cuts the batch.  Offsets,
tokens and values bit-exact; nothing written past the output; the flags
(invalid index, overflow) raised exactly when the oracle's batch has
them."""
import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, to_np

pytestmark = pytest.mark.gpu


def _ctx(edp):
    cfg = edp.make_config(64, (1, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16)
    return edp.Ring(cfg, action=False, reward=False, done=False)


@pytest.mark.parametrize("seed", range(24))
def test_random_packed_deliveries(edp_lib, seed):
    edp = edp_lib
    from oracle import llm
    rng = np.random.default_rng(7000 + seed)
    n_seq = int(rng.integers(1, 401))
    kind = rng.random(n_seq)
    lens = np.where(kind < 0.15, 0,
           np.where(kind < 0.45, rng.integers(1, 4, n_seq),
           np.where(kind < 0.9, rng.integers(4, 3000, n_seq),
                    rng.integers(4096, 9000, n_seq)))).astype(np.uint64)
    seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    src_shift = int(rng.integers(0, 4))  # the rollout's start within a 16-byte run
    total_src = int(seq_off[-1])
    tok_store = torch.full((total_src + 8,), 0, dtype=torch.int32, device="cuda")
    tokens = rng.integers(0, 152064, size=total_src, dtype=np.int32)
    d_tok = tok_store[src_shift:src_shift + total_src]
    d_tok.copy_(torch.from_numpy(tokens))
    B = int(rng.integers(1, 3001))
    idx = rng.integers(0, n_seq, size=B).astype(np.int64)
    bad = rng.random(B) < 0.02
    idx[bad] = rng.choice([-1, n_seq, n_seq + 5], size=int(bad.sum()))
    with_values = bool(rng.integers(0, 2))
    value = rng.standard_normal(n_seq).astype(np.float32)
    ref, ref_off, ref_v = llm.pack(tokens, seq_off, idx, value if with_values else None)
    n = len(ref)
    cap = n if rng.random() < 0.7 else int(rng.integers(0, n + 1))
    cap = max(cap, 1)  # out_cap counts elements available; at least one
    t_shift, v_shift = int(rng.integers(0, 4)), int(rng.integers(0, 4))
    base_t = torch.full((cap + 8,), -7, dtype=torch.int32, device="cuda")
    out = base_t[t_shift:t_shift + cap]
    ov = None
    if with_values:
        base_v = torch.full((cap + 8,), float("nan"), device="cuda")
        ov = base_v[v_shift:v_shift + cap]
    ooff = torch.full((B + 1,), -1, dtype=torch.int64, device="cuda")
    ring = _ctx(edp)
    edp.edp_pack_deliver(ring.ctx, d_tok, cuda(seq_off), n_seq, cuda(idx), B, out, ooff, cap,
                         seq_value=cuda(value) if with_values else None, out_value=ov)
    status, msg = edp.edp_sync_status(ring.ctx)
    assert (status != edp.EDP_OK) == (bool(bad.any()) or cap < n), (status, msg)
    assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
    w = min(cap, n)
    assert np.array_equal(to_np(out)[:w], ref[:w])
    assert (to_np(out)[w:] == -7).all()  # past the batch: untouched
    assert (to_np(base_t[:t_shift]) == -7).all() and (to_np(base_t[t_shift + cap:]) == -7).all()
    if with_values:
        assert np.array_equal(bits(ov)[:w], ref_v[:w].view(np.uint32))
        assert np.isnan(to_np(ov)[w:]).all()
        assert np.isnan(to_np(base_v[:v_shift])).all()
        assert np.isnan(to_np(base_v[v_shift + cap:])).all()
    ring.close()
