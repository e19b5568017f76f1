"""LLM post-training operators, written out from their definitions (test
infrastructure only: the tests and the benchmark's CPU leg may use it, the
library never).

Group-relative advantages (GRPO, Shao et al. 2024; advantage computation is
an ingestion step in the paper's post-training map, Appendix A): for the
responses of one prompt, A_i = (r_i - mean) / (std + eps), std the sample
standard deviation (divisor n - 1, 0 for one response), A = 0 where
std + eps = 0; fp64, rounded once to fp32.  Packed delivery: the selected
variable-length sequences concatenated in batch order, with offsets and a
per-sequence value repeated on each token.  Plain loops over groups and
sequences.
"""
import math

import numpy as np


def grpo_advantage(r, group_off, eps):
    r = np.asarray(r, np.float32)
    out = np.zeros(len(r), np.float32)
    for g in range(len(group_off) - 1):
        lo, hi = int(group_off[g]), int(group_off[g + 1])
        if hi <= lo:
            continue
        vals = [float(v) for v in r[lo:hi]]
        n = hi - lo
        mean = math.fsum(vals) / n
        var = math.fsum((v - mean) ** 2 for v in vals) / (n - 1) if n > 1 else 0.0
        den = math.sqrt(var) + float(np.float32(eps))
        for i, v in enumerate(vals):
            out[lo + i] = np.float32((v - mean) / den) if den > 0 else np.float32(0.0)
    return out


def pack(tokens, seq_off, idx, seq_value=None):
    """(out_tokens, out_off, out_value): sequence idx[k] after those before it;
    an index outside the sequences contributes nothing."""
    n_seq = len(seq_off) - 1
    parts, vals, off = [], [], [0]
    for s in idx:
        s = int(s)
        if 0 <= s < n_seq:
            seg = tokens[int(seq_off[s]):int(seq_off[s + 1])]
        else:
            seg = tokens[0:0]
        parts.append(seg)
        if seq_value is not None:
            vals.append(np.full(len(seg), seq_value[s] if 0 <= s < n_seq else 0,
                                np.float32))
        off.append(off[-1] + len(seg))
    out = np.concatenate(parts) if parts else np.zeros(0, np.int32)
    ov = np.concatenate(vals) if seq_value is not None and vals else None
    return out.astype(np.int32), np.array(off, np.uint64), ov
