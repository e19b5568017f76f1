"""Bandwidth-aware placement, written out from the paper (test
infrastructure only: the tests and the benchmark's CPU leg may use it, the
library never).

Sec. 5.1 models a placement's per-sample transfer latency as the actor ->
buffer leg plus the buffer -> learner leg, each size over effective
bandwidth; Eq. 1 (Sec. 5.2) takes the feasible minimum, found by the linear
scan of Alg. 1; Appendix D precomputes the choice over a range of sizes (the
placement map).  A two-tier placement reads a share h of the samples from
its first tier, h = min(1, Mem1 / (C_buf x)), the one-node analogue of the
paper's local / remote mixture.  Options are dicts: bw_in, bw_out, mem and,
for two tiers, bw_out2, mem2.
"""
import math


def transfer_latency(opt, c_buf, x):
    """T(p, x) = x / BW(actor -> p) + x / BW(p -> GPU); +inf when the buffer
    C_buf x does not fit the placement's memory (the constraint of Eq. 1)."""
    need = c_buf * x
    two = "bw_out2" in opt
    mem = opt["mem"] + opt["mem2"] if two else opt["mem"]
    if need > mem:
        return math.inf
    if not two:
        leg_out = x / opt["bw_out"]
    else:
        h = 1.0 if opt["mem"] >= need else opt["mem"] / need
        leg_out = x * (h / opt["bw_out"] + (1.0 - h) / opt["bw_out2"])
    return x / opt["bw_in"] + leg_out


def choose(opts, c_buf, x):
    """Alg. 1: scan the candidates, keep the feasible one with the smallest
    latency (strictly smaller replaces, so the first wins a tie); returns
    (index or len(opts) if none fits, latencies)."""
    best, t_min, ts = len(opts), math.inf, []
    for i, o in enumerate(opts):
        t = transfer_latency(o, c_buf, x)
        ts.append(t)
        if t < t_min:
            best, t_min = i, t
    return best, ts


def placement_map(opts, c_buf, xs):
    """Appendix D: the scan solved once per size."""
    return [choose(opts, c_buf, x)[0] for x in xs]
