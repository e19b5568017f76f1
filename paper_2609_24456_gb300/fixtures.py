"""Seeded synthetic inputs for the experience path.

This module only draws input data: transition payloads and metadata, rollout
signals and TD errors.  It holds none of the method's arithmetic (no
sampling, priority rule, transform, advantage or shuffle), so both the CUDA
path and the CPU oracle may consume what it produces.

Two kinds of generator:

* ``numpy`` draws (PCG64 keyed by ``(seed, stream)``) for inputs that fit in
  host memory: per-transition metadata, rollouts, TD errors, small payloads.
* a counter-based *content function* for payloads too large to keep on the
  host (GB-scale replay rings).  Word ``w`` of the payload of the transition
  with logical id ``L`` is ``content_word(seed, L, w)``, a 32-bit integer hash
  of (seed, L, w): two multiply/xor-shift rounds in the style of the
  integer-hash family of Wellons' "hash prospector".  Every intermediate
  product stays below 2^63, so the same values come out of numpy (host, for
  the oracle) and of torch int64 arithmetic (device, to fill rings quickly).
"""
import numpy as np

M32 = 0xFFFFFFFF
_C_ID, _C_W, _C_SEED, _C_OFF = 0x2545F491, 0x6C8E9CF5, 0x165667B1, 0x27D4EB2F
_C_MIX1, _C_MIX2 = 0x7FEB352D, 0x2C1B3C6D

# streams of the numpy generators
S_FRAMES, S_ACTION, S_REWARD, S_DONE, S_TD, S_OBS, S_VALUE, S_TOKENS = range(8)
S_LLM_LEN, S_LLM_TOK, S_LLM_REWARD = range(8, 11)


def rng(seed: int, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([int(seed), int(stream)]))


# --- replay transitions (Atari-like DQN workload) ----------------------------
def dqn_transitions(seed: int, n: int, frame_bytes: int = 84 * 84,
                    done_p: float = 0.01, with_frames: bool = True):
    """n transitions: uint8 frame (uniform bytes), int32 action in [0, 6),
    fp32 reward in {-1, 0, 1} with p = (0.1, 0.8, 0.1), uint8 done ~
    Bernoulli(done_p)."""
    frames = (rng(seed, S_FRAMES).integers(0, 256, size=(n, frame_bytes),
                                           dtype=np.uint8)
              if with_frames else None)
    action = rng(seed, S_ACTION).integers(0, 6, size=n).astype(np.int32)
    reward = rng(seed, S_REWARD).choice(
        np.array([-1.0, 0.0, 1.0], np.float32), size=n,
        p=[0.1, 0.8, 0.1]).astype(np.float32)
    done = (rng(seed, S_DONE).random(n) < done_p).astype(np.uint8)
    return frames, action, reward, done


def td_errors(seed: int, n: int, round_: int = 0) -> np.ndarray:
    """Fresh TD errors delta ~ Exp(1), fp32."""
    g = np.random.Generator(np.random.PCG64([int(seed), S_TD, int(round_)]))
    return g.exponential(1.0, size=n).astype(np.float32)


# --- on-policy rollout (PPO workload) -----------------------------------------
def ppo_rollout(seed: int, T: int, E: int, H: int = 64, W: int = 64,
                C: int = 3, done_p: float = 0.005, with_obs: bool = True):
    """T steps of E environments, time-major: obs [T*E, H*W*C] uint8 HWC
    (uniform), reward [T, E] fp32 N(0, 1), value [T+1, E] fp32 N(0, 1),
    done [T, E] uint8 ~ Bernoulli(done_p)."""
    obs = (rng(seed, S_OBS).integers(0, 256, size=(T * E, H * W * C),
                                     dtype=np.uint8) if with_obs else None)
    r = rng(seed, S_REWARD).standard_normal((T, E)).astype(np.float32)
    v = rng(seed, S_VALUE).standard_normal((T + 1, E)).astype(np.float32)
    d = (rng(seed, S_DONE).random((T, E)) < done_p).astype(np.uint8)
    return obs, r, v, d


# --- multimodal payload (image + tokens) --------------------------------------
def mm_metadata(seed: int, n: int, tokens: int = 512, vocab: int = 32000):
    """tokens [n, L] int32 uniform in [0, vocab), reward [n] fp32 N(0, 1)."""
    tok = rng(seed, S_TOKENS).integers(0, vocab, size=(n, tokens),
                                       dtype=np.int32) if tokens else None
    rew = rng(seed, S_REWARD).standard_normal(n).astype(np.float32)
    return tok, rew


# --- counter-based content function -------------------------------------------
def content_words(seed: int, ids, nwords: int) -> np.ndarray:
    """uint32 [len(ids), nwords]: payload words of the given logical ids."""
    ids = np.asarray(ids, dtype=np.uint64).reshape(-1, 1)
    w = np.arange(nwords, dtype=np.uint64).reshape(1, -1)
    m = np.uint64(M32)
    x = (((ids & m) * np.uint64(_C_ID)) & m) + ((w * np.uint64(_C_W)) & m)
    x = (x + np.uint64((int(seed) * _C_SEED + _C_OFF) & M32)) & m
    x ^= x >> np.uint64(16)
    x = (x * np.uint64(_C_MIX1)) & m
    x ^= x >> np.uint64(15)
    x = (x * np.uint64(_C_MIX2)) & m
    x ^= x >> np.uint64(16)
    return x.astype(np.uint32)


def content_bytes(seed: int, ids, nbytes: int) -> np.ndarray:
    """uint8 [len(ids), nbytes] (nbytes % 4 == 0), little-endian words."""
    assert nbytes % 4 == 0
    return np.ascontiguousarray(content_words(seed, ids, nbytes // 4)).view(
        np.uint8).reshape(-1, nbytes)


def content_fill_torch(seed: int, first_id: int, out):
    """Fill a device tensor ``out`` (any dtype, shape [n, ...], row bytes a
    multiple of 4) with the content of logical ids first_id .. first_id+n-1,
    using torch int64 arithmetic on out's device."""
    import torch
    n = out.shape[0]
    nbytes = out[0].numel() * out.element_size() if n else 0
    assert nbytes % 4 == 0
    nwords = nbytes // 4
    dev = out.device
    words = out.view(n, -1).view(torch.int32) if n else None
    # bound the int64 temporaries to ~256 Mi elements per chunk
    rows = max(1, (1 << 28) // max(nwords, 1))
    for r0 in range(0, n, rows):
        r1 = min(n, r0 + rows)
        ids = torch.arange(first_id + r0, first_id + r1, device=dev,
                           dtype=torch.int64).view(-1, 1)
        w = torch.arange(nwords, device=dev, dtype=torch.int64).view(1, -1)
        x = ((ids & M32) * _C_ID) & M32
        x = x + ((w * _C_W) & M32)
        x = (x + ((int(seed) * _C_SEED + _C_OFF) & M32)) & M32
        x ^= x >> 16
        x = (x * _C_MIX1) & M32
        x ^= x >> 15
        x = (x * _C_MIX2) & M32
        x ^= x >> 16
        x = torch.where(x >= (1 << 31), x - (1 << 32), x)
        words[r0:r1].copy_(x.to(torch.int32))
    return out


def token_content(seed: int, ids, tokens: int, vocab: int = 32000):
    """int32 [len(ids), tokens] token ids in [0, vocab) from the content
    function (stream of seed + 7919, so it differs from the image words)."""
    return (content_words(seed + 7919, ids, tokens) % np.uint32(vocab)).astype(
        np.int32)


def token_fill_torch(seed: int, first_id: int, out, vocab: int = 32000):
    import torch
    content_fill_torch(seed + 7919, first_id, out)
    u = out.to(torch.int64) & M32
    out.copy_((u % vocab).to(torch.int32))
    return out


# --- LLM post-training batch (GRPO) -------------------------------------------
def llm_rollout(seed: int, n_prompts: int, group: int, lmin: int = 128,
                lmax: int = 4096, vocab: int = 152064, binary_frac: float = 0.5):
    """A GRPO batch: n_prompts groups of `group` responses with lengths
    U[lmin, lmax] tokens, token ids U[0, vocab) (int32, packed, with uint64
    offsets), and one reward per response: for a share binary_frac of the
    groups 0/1 correctness ~ Bernoulli(0.4) (math RL; some groups constant),
    for the others N(0, 1).  Returns tokens, seq_off, rewards, group_off."""
    n = n_prompts * group
    lens = rng(seed, S_LLM_LEN).integers(lmin, lmax + 1, size=n).astype(np.uint64)
    seq_off = np.zeros(n + 1, np.uint64)
    np.cumsum(lens, out=seq_off[1:])
    tokens = rng(seed, S_LLM_TOK).integers(0, vocab, size=int(seq_off[-1]),
                                           dtype=np.int32)
    g = rng(seed, S_LLM_REWARD)
    binary = g.random(n_prompts) < binary_frac
    r = np.where(np.repeat(binary, group), (g.random(n) < 0.4).astype(np.float32),
                 g.standard_normal(n).astype(np.float32)).astype(np.float32)
    group_off = (np.arange(n_prompts + 1, dtype=np.uint64) * np.uint64(group))
    return tokens, seq_off, r, group_off
