"""GPU parity of the LLM post-training operators through the C ABI:
group-relative advantages within 1 ulp of the fp64 oracle (rounded once to
fp32), packed delivery of variable-length sequences bit-exact (tokens,
offsets, per-token values), including groups of one, constant groups,
repeated and invalid indices and an output buffer that is too small, at
small sizes and at a 512-prompt x 16-response batch."""
import numpy as np
import pytest
import torch

from gpu_util import bits, cuda, fx, to_np

pytestmark = pytest.mark.gpu


def _ctx(edp):
    cfg = edp.make_config(64, (1, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16)
    return edp.Ring(cfg, action=False, reward=False, done=False)


def _ulps(a, b):
    a = a.view(np.int32).astype(np.int64)
    b = b.view(np.int32).astype(np.int64)
    return np.abs(a - b)


def _grpo_check(edp, ring, r, goff, eps):
    d_r, d_off = cuda(r), cuda(goff)
    adv = torch.full((len(r),), float("nan"), device="cuda")
    edp.edp_grpo_advantage(ring.ctx, d_r, d_off, len(goff) - 1, eps, adv)
    edp.edp_sync(ring.ctx)
    from oracle import llm
    ref = llm.grpo_advantage(r, goff, eps)
    got = to_np(adv)
    assert _ulps(got, ref).max() <= 1
    return got, ref


def test_grpo_edge_groups(edp_lib):
    edp = edp_lib
    ring = _ctx(edp)
    r = np.array([1, 2, 3, 5, 5, 5, 7, 0, 1, 4], np.float32)
    goff = np.array([0, 3, 6, 7, 9, 9, 10], np.uint64)  # includes an empty group
    got, _ = _grpo_check(edp, ring, r, goff, 0.0)
    assert list(got[:7]) == [-1.0, 0.0, 1.0, 0.0, 0.0, 0.0, 0.0]
    assert got[9] == 0.0  # a group of one
    _grpo_check(edp, ring, r, goff, 1e-6)


@pytest.mark.parametrize("group", [1, 2, 7, 16, 33, 1000])
def test_grpo_random(edp_lib, group):
    edp = edp_lib
    ring = _ctx(edp)
    _, _, r, goff = fx.llm_rollout(group, 300, group, lmin=1, lmax=2)
    _grpo_check(edp, ring, r, goff, 1e-6)


def _pack_check(edp, ring, tokens, seq_off, idx, value, cap=None):
    from oracle import llm
    ref, ref_off, ref_v = llm.pack(tokens, seq_off, idx, value)
    cap = len(ref) if cap is None else cap
    B = len(idx)
    out = torch.full((max(cap, 1),), -7, dtype=torch.int32, device="cuda")
    ov = torch.full((max(cap, 1),), float("nan"), device="cuda")
    ooff = torch.full((B + 1,), -1, dtype=torch.int64, device="cuda")
    d_tok, d_off, d_idx, d_v = cuda(tokens), cuda(seq_off), cuda(np.asarray(idx, np.int64)), \
        cuda(value)
    edp.edp_pack_deliver(ring.ctx, d_tok, d_off, len(seq_off) - 1, d_idx, B, out, ooff, cap,
                         seq_value=d_v, out_value=ov)
    return ref, ref_off, ref_v, out, ooff, ov


def test_pack_small_ragged(edp_lib):
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, _ = fx.llm_rollout(4, 10, 4, lmin=0, lmax=700)  # empty ones too
    rng = np.random.default_rng(5)
    for B in [1, 3, 40, 1500]:
        idx = rng.integers(0, 40, size=B)
        ref, ref_off, ref_v, out, ooff, ov = _pack_check(edp, ring, tokens, seq_off, idx, r)
        edp.edp_sync(ring.ctx)
        n = len(ref)
        assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
        assert np.array_equal(to_np(out)[:n], ref)
        assert np.array_equal(bits(ov)[:n], ref_v.view(np.uint32))


@pytest.mark.parametrize("B", [65536, 65537, 70000])
def test_pack_many_chunks(edp_lib, B):
    """Batches around the size where the chunk prefixes move from the gather
    CTAs to the lengths pass (256 chunks of 256 entries)."""
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, _ = fx.llm_rollout(9, 500, 2, lmin=0, lmax=9)
    idx = np.random.default_rng(B).integers(0, 1000, size=B)
    ref, ref_off, ref_v, out, ooff, ov = _pack_check(edp, ring, tokens, seq_off, idx, r)
    edp.edp_sync(ring.ctx)
    n = len(ref)
    assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
    assert np.array_equal(to_np(out)[:n], ref)
    assert np.array_equal(bits(ov)[:n], ref_v.view(np.uint32))


@pytest.mark.parametrize("tok_shift,val_shift", [(1, 2), (3, 0), (2, 3)])
def test_pack_unaligned_outputs(edp_lib, tok_shift, val_shift):
    """Output arrays starting 4, 8 or 12 bytes past a 16-byte boundary (each
    its own offset), with sequences of every length 0..200 from every
    source alignment: the vector body, the token-by-token ends and the
    value fill all land where the oracle puts them."""
    edp = edp_lib
    ring = _ctx(edp)
    from oracle import llm
    lens = np.arange(0, 201, dtype=np.uint64)
    seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    rng = np.random.default_rng(tok_shift * 7 + val_shift)
    tokens = rng.integers(0, 152064, size=int(seq_off[-1]), dtype=np.int32)
    value = rng.standard_normal(len(lens)).astype(np.float32)
    idx = rng.permutation(len(lens)).astype(np.int64)
    ref, ref_off, ref_v = llm.pack(tokens, seq_off, idx, value)
    n = len(ref)
    base_t = torch.full((n + 8,), -7, dtype=torch.int32, device="cuda")
    base_v = torch.full((n + 8,), float("nan"), device="cuda")
    out, ov = base_t[tok_shift:tok_shift + n], base_v[val_shift:val_shift + n]
    assert out.data_ptr() % 16 == 4 * tok_shift and ov.data_ptr() % 16 == 4 * val_shift
    ooff = torch.full((len(idx) + 1,), -1, dtype=torch.int64, device="cuda")
    edp.edp_pack_deliver(ring.ctx, cuda(tokens), cuda(seq_off), len(lens), cuda(idx),
                         len(idx), out, ooff, n, seq_value=cuda(value), out_value=ov)
    edp.edp_sync(ring.ctx)
    assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
    assert np.array_equal(to_np(out), ref)
    assert np.array_equal(bits(ov), ref_v.view(np.uint32))
    # nothing written outside the output
    assert (to_np(base_t[:tok_shift]) == -7).all() and (to_np(base_t[tok_shift + n:]) == -7).all()
    assert np.isnan(to_np(base_v[:val_shift])).all() and np.isnan(to_np(base_v[val_shift + n:])).all()


@pytest.mark.parametrize("shift", [0, 1, 3])
def test_pack_long_sequences(edp_lib, shift):
    """Sequences longer than one 4,096-token bulk copy (4,095 .. 10,000
    tokens, several chunks each) among short ones, from sources at every
    alignment, into an output starting 0, 4 or 12 bytes past a 16-byte
    boundary; then the same batch cut by out_cap inside the second chunk of
    a long sequence."""
    edp = edp_lib
    ring = _ctx(edp)
    from oracle import llm
    lens = np.array([4095, 1, 4096, 3, 4097, 5, 8191, 2, 8192, 10000, 0, 7], np.uint64)
    seq_off = np.concatenate([[0], np.cumsum(lens)]).astype(np.uint64)
    rng = np.random.default_rng(40 + shift)
    tokens = rng.integers(0, 152064, size=int(seq_off[-1]), dtype=np.int32)
    value = rng.standard_normal(len(lens)).astype(np.float32)
    idx = np.concatenate([rng.permutation(len(lens)), [9, 6]]).astype(np.int64)
    ref, ref_off, ref_v = llm.pack(tokens, seq_off, idx, value)
    n = len(ref)
    for cap in (n, int(ref_off[list(idx).index(9)]) + 4096 + 1001):
        base_t = torch.full((n + 8,), -7, dtype=torch.int32, device="cuda")
        base_v = torch.full((n + 8,), float("nan"), device="cuda")
        out, ov = base_t[shift:shift + cap], base_v[shift:shift + cap]
        ooff = torch.full((len(idx) + 1,), -1, dtype=torch.int64, device="cuda")
        edp.edp_pack_deliver(ring.ctx, cuda(tokens), cuda(seq_off), len(lens), cuda(idx),
                             len(idx), out, ooff, cap, seq_value=cuda(value), out_value=ov)
        if cap < n:
            with pytest.raises(edp.EdpError) as e:
                edp.edp_sync(ring.ctx)
            assert str(n) in str(e.value)
        else:
            edp.edp_sync(ring.ctx)
        assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
        assert np.array_equal(to_np(out), ref[:cap])
        assert np.array_equal(bits(ov), ref_v[:cap].view(np.uint32))
        # nothing written past the output or before it
        assert (to_np(base_t[:shift]) == -7).all() and (to_np(base_t[shift + cap:]) == -7).all()
        assert np.isnan(to_np(base_v[:shift])).all() and np.isnan(to_np(base_v[shift + cap:])).all()


def test_pack_invalid_index_and_overflow(edp_lib):
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, _ = fx.llm_rollout(6, 4, 2, lmin=5, lmax=50)
    idx = [3, -1, 8, 2]  # -1 and 8 are outside the 8 sequences
    ref, ref_off, ref_v, out, ooff, ov = _pack_check(edp, ring, tokens, seq_off, idx, r)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_sync(ring.ctx)
    assert e.value.status == edp.EDP_ERR_INVALID
    n = len(ref)
    assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
    assert np.array_equal(to_np(out)[:n], ref)
    # output buffer too small: the first `cap` elements are written, the
    # rest are not, and the error names the size needed
    idx = [0, 1, 2, 3, 4, 5]
    from oracle import llm
    full, full_off, full_v = llm.pack(tokens, seq_off, idx, r)
    cap = len(full) - 17
    ref, ref_off, ref_v, out, ooff, ov = _pack_check(edp, ring, tokens, seq_off, idx, r, cap)
    with pytest.raises(edp.EdpError) as e:
        edp.edp_sync(ring.ctx)
    assert str(len(full)) in str(e.value)
    assert np.array_equal(to_np(ooff).view(np.uint64), full_off)
    assert np.array_equal(to_np(out)[:cap], full[:cap])
    assert np.array_equal(bits(ov)[:cap], full_v[:cap].view(np.uint32))
    edp.edp_sync(ring.ctx)  # the flag was cleared


def test_grpo_batch_full_size(edp_lib):
    """512 prompts x 16 responses of 128..4,096 tokens (about 17 M tokens):
    advantages, then the whole batch delivered in a shuffled order with
    every token carrying its response's advantage."""
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, goff = fx.llm_rollout(7, 512, 16)
    n = len(r)
    adv_got, adv_ref = _grpo_check(edp, ring, r, goff, 1e-6)
    perm = np.random.default_rng(8).permutation(n)
    ref, ref_off, ref_v, out, ooff, ov = _pack_check(edp, ring, tokens, seq_off, perm,
                                                     adv_got)
    edp.edp_sync(ring.ctx)
    assert np.array_equal(to_np(ooff).view(np.uint64), ref_off)
    assert np.array_equal(to_np(out), ref)
    assert np.array_equal(bits(ov), ref_v.view(np.uint32))


@pytest.mark.parametrize("case", ["full", "ragged_invalid", "no_values"])
def test_grpo_pack_fused(edp_lib, case):
    """edp_grpo_pack_deliver against the two calls it fuses (bit for bit:
    advantages, tokens, offsets, per-token values) and the oracle, on the
    512 x 16 batch and on a small ragged one with an index out of range."""
    edp = edp_lib
    ring = _ctx(edp)
    from oracle import llm
    if case == "full":
        tokens, seq_off, r, goff = fx.llm_rollout(11, 512, 16)
        idx = np.random.default_rng(12).permutation(len(r)).astype(np.int64)
    else:
        tokens, seq_off, r, goff = fx.llm_rollout(13, 9, 5, lmin=0, lmax=300)
        idx = np.random.default_rng(14).integers(0, len(r), size=700).astype(np.int64)
        if case == "ragged_invalid":
            idx[[3, 500]] = [-2, len(r)]
    n, B = len(r), len(idx)
    adv_ref = llm.grpo_advantage(r, goff, 1e-6)
    d_r, d_goff, d_tok, d_off, d_idx = cuda(r), cuda(goff), cuda(tokens), cuda(seq_off), \
        cuda(idx)
    total = int(sum(int(seq_off[s + 1] - seq_off[s]) for s in idx if 0 <= s < n))
    outs = []
    for fused in (False, True):
        adv = torch.full((n,), float("nan"), device="cuda")
        out = torch.full((max(total, 1),), -7, dtype=torch.int32, device="cuda")
        ov = torch.full((max(total, 1),), float("nan"), device="cuda")
        oo = torch.full((B + 1,), -1, dtype=torch.int64, device="cuda")
        vals = None if case == "no_values" else ov
        if fused:
            edp.edp_grpo_pack_deliver(ring.ctx, d_r, d_goff, len(goff) - 1, 1e-6, adv, d_tok,
                                      d_off, n, d_idx, B, out, oo, total, out_value=vals)
        else:
            edp.edp_grpo_advantage(ring.ctx, d_r, d_goff, len(goff) - 1, 1e-6, adv)
            edp.edp_pack_deliver(ring.ctx, d_tok, d_off, n, d_idx, B, out, oo, total,
                                 seq_value=None if vals is None else adv, out_value=vals)
        status, _ = edp.edp_sync_status(ring.ctx)
        assert status == (edp.EDP_ERR_INVALID if case == "ragged_invalid" else edp.EDP_OK)
        outs.append((bits(adv), to_np(out), to_np(oo), bits(ov)))
    for x, y in zip(*outs):
        assert np.array_equal(x, y)
    assert _ulps(outs[1][0].view(np.float32), adv_ref).max() <= 1
    ref, ref_off, ref_v = llm.pack(tokens, seq_off, idx, outs[1][0].view(np.float32))
    assert np.array_equal(outs[1][2].view(np.uint64), ref_off)
    assert np.array_equal(outs[1][1][:len(ref)], ref)
    if case != "no_values":
        assert np.array_equal(outs[1][3][:len(ref)], ref_v.view(np.uint32))


def test_grpo_pack_fused_argument_errors(edp_lib):
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, goff = fx.llm_rollout(15, 4, 3, lmin=1, lmax=20)
    n = len(r)
    d = dict(r=cuda(r), goff=cuda(goff), tok=cuda(tokens), off=cuda(seq_off),
             idx=cuda(np.arange(n, dtype=np.int64)))
    adv = torch.empty(n, device="cuda")
    out = torch.empty(int(seq_off[-1]), dtype=torch.int32, device="cuda")
    oo = torch.empty(n + 1, dtype=torch.int64, device="cuda")

    def call(**kw):
        a = dict(r=d["r"], goff=d["goff"], ng=len(goff) - 1, eps=1e-6, adv=adv,
                 tok=d["tok"], off=d["off"], nseq=n, idx=d["idx"], B=n, out=out, oo=oo)
        a.update(kw)
        edp.edp_grpo_pack_deliver(ring.ctx, a["r"], a["goff"], a["ng"], a["eps"], a["adv"],
                                  a["tok"], a["off"], a["nseq"], a["idx"], a["B"], a["out"],
                                  a["oo"], int(seq_off[-1]))

    call()
    edp.edp_sync(ring.ctx)
    for kw in (dict(ng=0), dict(eps=-1.0), dict(eps=float("nan")), dict(adv=None),
               dict(idx=None), dict(B=0), dict(nseq=0), dict(B=(1 << 20) + 1),
               dict(tok=torch.from_numpy(tokens))):  # host memory, not device
        with pytest.raises(edp.EdpError) as e:
            call(**kw)
        assert e.value.status == edp.EDP_ERR_INVALID, kw


def test_pack_into_host_outputs(edp_lib):
    """Packed tokens, offsets and per-token values written straight into
    page-locked host memory equal the device-output delivery."""
    edp = edp_lib
    ring = _ctx(edp)
    tokens, seq_off, r, goff = fx.llm_rollout(17, 20, 4, lmin=0, lmax=500)
    idx = np.random.default_rng(18).permutation(len(r)).astype(np.int64)
    n, B = len(r), len(idx)
    total = int(seq_off[-1])
    d_args = (cuda(r), cuda(goff), len(goff) - 1, 1e-6)
    res = []
    for host in (False, True):
        mk = (lambda shape, dt: torch.empty(shape, dtype=dt, pin_memory=True)) if host else \
             (lambda shape, dt: torch.empty(shape, dtype=dt, device="cuda"))
        adv = torch.empty(n, device="cuda")
        out, oo, ov = mk(total, torch.int32), mk(B + 1, torch.int64), mk(total, torch.float32)
        edp.edp_grpo_pack_deliver(ring.ctx, *d_args, adv, cuda(tokens), cuda(seq_off), n,
                                  cuda(idx), B, out, oo, total, out_value=ov)
        edp.edp_sync(ring.ctx)
        res.append((to_np(out), to_np(oo), bits(ov)))
    for x, y in zip(*res):
        assert np.array_equal(x, y)
