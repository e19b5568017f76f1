#!/usr/bin/env python3
"""Benchmark of the experience-path hot path on one GB300 (or N replicas).

Default workload (the largest HBM-resident configuration): multimodal
replay over 200,000 transitions of a uint8 3x224x224 image, 512 int32
tokens and a reward (~30.5 GB in HBM), uniform batch 1,024 delivered as
per-channel normalised bf16 with collated tokens and rewards.  One step =
one round of the hot path: the uniform draw and the fused gather +
normalise + collate.  Other workloads (--workload): prioritized replay over
1,000,000 84x84 frames (per1m: stratified sampling through the sum-tree,
frame-stack delivery of obs and next_obs as fp32 with importance weights,
priority update), the tiny DQN replay, the PPO iteration, the two-tier ring
beyond HBM and the GRPO batch.

Prints ONE JSON line (rank 0).  `value` = delivered GB/s (algorithmic bytes
of the rounds / device time), `e2e` = the same through the C ABI with host
buffers (inputs copied in and the learner batch written to host memory
every step).

--impl reference times the CPU oracle (plain C, all host cores) on the same
workload and metric; each step is one round of the same per-round work.
"""
import argparse
import ctypes

import numpy as np
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

HBM_FALLBACK_GBS = 6800.0
ALPHA, EPS, BETA = 0.6, 1e-6, 0.4


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(p))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return HBM_FALLBACK_GBS, "fallback"


# ----------------------------------------------------------------------------
# clocks during the timed region: NVML poller (1 ms) + nvidia-smi (100 ms)
# ----------------------------------------------------------------------------
REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting",
           0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
           0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
           0x100: "display_clock_setting"}


class Clocks:
    def __init__(self, cuda_index):
        self.samples = []
        self.max_mhz = None
        self._stop = threading.Event()
        self._nvml = None
        self._smi = None
        self._smi_file = None
        try:
            import torch
            props = torch.cuda.get_device_properties(cuda_index)
            bus = "%08x:%02x:%02x.0" % (getattr(props, "pci_domain_id", 0),
                                        props.pci_bus_id, props.pci_device_id)
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise OSError("nvmlInit")
            h = ctypes.c_void_p()
            if nv.nvmlDeviceGetHandleByPciBusId_v2(bus.encode(), ctypes.byref(h)) != 0:
                raise OSError("nvml handle")
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = float(mx.value)
            self._nvml = (nv, h)
            self._bus = bus
        except Exception:
            self._nvml = None

    def _poll(self):
        nv, h = self._nvml
        mhz = ctypes.c_uint()
        rs = ctypes.c_ulonglong()
        get_r = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(mhz)) == 0:
                r = rs.value if get_r(h, ctypes.byref(rs)) == 0 else 0
                self.samples.append((float(mhz.value), int(r)))
            time.sleep(0.001)

    def start(self):
        if self._nvml:
            self._t = threading.Thread(target=self._poll, daemon=True)
            self._t.start()
        try:
            self._smi_file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                 "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                 "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
            self._smi = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + q, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=self._smi_file, stderr=subprocess.DEVNULL)
        except Exception:
            self._smi = None

    def stop(self):
        self._stop.set()
        if self._nvml:
            self._t.join(timeout=1)
        smi = []
        if self._smi:
            self._smi.terminate()
            try:
                self._smi.wait(timeout=2)
            except Exception:
                self._smi.kill()
            try:
                self._smi_file.flush()
                for line in open(self._smi_file.name):
                    f = [x.strip() for x in line.split(",")]
                    if len(f) >= 9:
                        smi.append(f)
                os.unlink(self._smi_file.name)
            except Exception:
                pass
        out = {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [],
               "samples": len(self.samples), "smi_samples": len(smi)}
        if self.samples:
            out["sm_mhz"] = statistics.median(s[0] for s in self.samples)
            bits = 0
            for _, r in self.samples:
                bits |= r
            out["reasons"] = sorted(n for b, n in REASONS.items()
                                    if bits & b and n != "gpu_idle")
        elif smi:
            try:
                out["sm_mhz"] = statistics.median(float(f[1]) for f in smi)
                out["sm_max_mhz"] = float(smi[0][2])
                names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                         "sw_power_cap"]
                out["reasons"] = sorted({names[i] for f in smi for i in range(4)
                                         if f[5 + i].lower() == "active"})
            except Exception:
                pass
        return out


# ----------------------------------------------------------------------------
# helpers
# ----------------------------------------------------------------------------
def kernel_traffic(kernel, workload):
    """Per-launch DRAM bytes from the committed ncu summary, or None when the
    kernel source changed since the counters were taken."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    try:
        d = json.load(open(p))[kernel]
    except Exception:
        return None
    src = os.path.join(ROOT, "paper_2609_24456_gb300", "csrc", d["source"])
    try:
        h = hashlib.sha256(open(src, "rb").read()).hexdigest()
    except OSError:
        return None
    if h != d.get("source_sha256") or d.get("workload") != workload:
        return None
    return d.get("dram_bytes_per_launch")


def dev(a, device):
    import numpy as np
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint32:
        a = a.view(np.int32)
    return torch.from_numpy(a).to(device)


def oracle_set_threads(n):
    import oracle
    L = oracle.lib()
    L.orc_set_threads.argtypes = [ctypes.c_int]
    L.orc_set_threads(int(n))


def oracle_threads():
    import oracle
    L = oracle.lib()
    try:
        fn = L.orc_num_threads
        fn.restype = ctypes.c_int
        return int(fn())
    except AttributeError:
        return os.cpu_count() or 1


# ----------------------------------------------------------------------------
# Workloads.  A workload fixes the synthetic data, the step (one pass of its
# hot path), the algorithmic bytes of a step and of its dominant kernel, the
# end-to-end user path and the oracle's bounded CPU sample.
# ----------------------------------------------------------------------------
class Workload:
    name = kernel = ""
    dtype = ""
    launches_per_round = 0
    # launches per round of schedules that differ from launches_per_round
    launches_by_schedule = {}
    h2d = d2h = 0

    def config(self):
        return {"workload": self.name}

    def schedules(self):
        """[(name, round function, description)], the main schedule first;
        every schedule runs the same work per round."""
        return [("one stream", self.round, "one stream")]

    def join(self):
        """Make the current stream wait for the workload's side streams."""
        import torch
        if getattr(self, "side_used", False):
            for st in self.sides:
                torch.cuda.current_stream().wait_stream(st)
        self.side_used = False
        self.in_flight = set()

    def _init_overlap(self, device, sets, sides=2):
        import torch
        self.sides = [torch.cuda.Stream(device=device) for _ in range(sides)]
        self.ready = [torch.cuda.Event() for _ in range(sets)]
        self.consumed = [torch.cuda.Event() for _ in range(sets)]
        self.in_flight = set()  # output sets whose delivery is not yet joined
        self.side_used = False

    def _overlapped(self, k, sample, deliver, after=None):
        """One round with its delivery on a side stream: sample() on the
        current stream; deliver(stream) on side stream k mod (number of side
        streams) once the sampling has finished; after() (if any) on the
        current stream meanwhile.  Consecutive deliveries alternate between
        the side streams, so one's ramp-up overlaps the previous one's tail.
        Output set k is reused only after its previous delivery has read
        its indices."""
        import torch
        main = torch.cuda.current_stream()
        if k in self.in_flight:
            main.wait_event(self.consumed[k])
        sample()
        self.ready[k].record()
        side = self.sides[k % len(self.sides)]
        with torch.cuda.stream(side):
            side.wait_event(self.ready[k])
            deliver(side)
            self.consumed[k].record()
        self.in_flight.add(k)
        self.side_used = True
        if after is not None:
            after()

    def _graph_or_eager(self, body, graph):
        import torch
        body()
        torch.cuda.synchronize()
        if not graph:
            return body
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="thread_local"):
            body()
        g.replay()
        torch.cuda.synchronize()
        return g.replay

    def time_deliver(self, n, mk, stream, graph=True):
        """Average duration (us) of the dominant kernel launched n times back
        to back (events bracket the launches; inputs are real batches)."""
        import torch
        run = self._graph_or_eager(lambda: [self.deliver_once(r) for r in range(n)],
                                   graph)
        e0, e1 = mk(), mk()
        e0.record(stream)
        run()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / n

    def time_calls(self, fn, n, mk, stream):
        """Average device time (us) of fn() run n times back to back from a
        CUDA graph (two eager calls first)."""
        import torch
        run = self._graph_or_eager(lambda: [fn() for _ in range(n)], True)
        e0, e1 = mk(), mk()
        e0.record(stream)
        run()
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) * 1e3 / n

    def time_latency(self, n, mk, stream):
        """Sample -> batch latency (us) of n steps: the time on the device
        from an event before the step's first call to one after its batch
        is complete.  Each step is queued behind a short spin kernel, so the
        host has submitted all of the step before the device reaches it:
        the events time the step's kernels and their launches, not the
        host's submission of the calls (nor the event nodes of a graph,
        which split it)."""
        import torch
        out = []
        for r in range(n):
            e0, e1 = mk(), mk()
            torch.cuda._sleep(200000)  # ~0.1 ms at 2 GHz: the host queues the step meanwhile
            e0.record(stream)
            self.latency_step(100000 + r, e1)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) * 1e3)
        return out


def _stack_bytes(B, K, F, next_obs=True):
    """Fused frame-stack delivery: unique frame reads (K+1 per sample with
    next_obs), fp32 writes of obs (+ next_obs), collate and IS scalars (idx
    8, q 4 read; isw 4, action 4, reward 4, done 1 written; action 4,
    reward 4, done K+1 read)."""
    frames = K + 1 if next_obs else K
    return B * (frames * F + (2 if next_obs else 1) * K * F * 4 + 33 + frames)


class PerReplay(Workload):
    """Prioritized replay: 1,000,000 uint8 84x84 frames (~7.06 GB), batch
    512, frame stack 4, obs + next_obs fp32, PER alpha 0.6 / beta 0.4 with
    priorities from Exp(1) TD errors; step = sample, deliver, update."""
    name = "per-replay-1M-84x84-B512"
    kernel = "k_deliver_stack_staged"
    dtype = "u8->f32"
    launches_per_round = 3

    def __init__(self, capacity=1_000_000, batch=512, K=4, seed=1235,
                 out_sets=4):
        self.cap, self.B, self.K, self.seed = capacity, batch, K, seed
        self.F = 84 * 84
        self.R = out_sets
        D = 1
        while 32 ** D < capacity:
            D += 1
        self.D = D
        B = batch
        self.deliver_bytes = _stack_bytes(B, K, self.F)
        # sampling: one 32-child row per global level + the leaf row, writes
        # idx and q
        self.sample_bytes = B * (32 * 8 * max(D - 3, 0) + 32 * 4 + 12)
        # update: idx, td, leaf read + write, D ancestors read + write (8 B)
        self.update_bytes = B * (8 + 4 + 8 + 16 * D)
        self.round_bytes = self.deliver_bytes + self.sample_bytes + self.update_bytes

    def config(self):
        return {"workload": self.name, "capacity": self.cap, "batch": self.B,
                "frame": "uint8 84x84", "frame_stack": self.K,
                "outputs": "obs+next_obs fp32 [B,4,84,84], action, reward, done, isw",
                "priorities": "PER alpha 0.6 (u32, 2^20 fixed point), beta 0.4",
                "l2": "ring %.2f GB > L2; outputs rotate over %d buffers (%.0f MB)"
                      % (self.cap * self.F / 1e9, self.R,
                         self.R * self.B * 2 * self.K * self.F * 4 / 1e6)}

    def setup(self, device):
        import torch
        from paper_2609_24456_gb300 import edp
        from paper_2609_24456_gb300 import fixtures as fx
        self.edp = edp
        cfg = edp.make_config(self.cap, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                              frame_stack=self.K, next_obs=True, prioritized=True,
                              device=device.index or 0)
        self.ring = edp.Ring(cfg)
        ctx = self.ring.ctx
        _, action, reward, done = fx.dqn_transitions(self.seed, self.cap,
                                                     with_frames=False)
        td = fx.td_errors(self.seed, self.cap)
        chunk = 65536
        staging = torch.empty((chunk, self.F), dtype=torch.uint8, device=device)
        qbuf = torch.empty(chunk, dtype=torch.int32, device=device)
        for lo in range(0, self.cap, chunk):
            hi = min(self.cap, lo + chunk)
            n = hi - lo
            fx.content_fill_torch(self.seed, lo, staging[:n])
            edp.edp_priorities_from_td(ctx, dev(td[lo:hi], device), n, ALPHA, EPS, qbuf)
            edp.edp_ingest(ctx, staging[:n], n, action=dev(action[lo:hi], device),
                           reward=dev(reward[lo:hi], device),
                           done=dev(done[lo:hi], device), q=qbuf)
        del staging
        edp.edp_sync(ctx)
        B, K, F = self.B, self.K, self.F
        self.outs = []
        for _ in range(self.R):
            o = dict(idx=torch.empty(B, dtype=torch.int64, device=device),
                     q=torch.empty(B, dtype=torch.int32, device=device),
                     obs=torch.empty((B, K, F), device=device),
                     nxt=torch.empty((B, K, F), device=device),
                     act=torch.empty(B, dtype=torch.int32, device=device),
                     rew=torch.empty(B, device=device),
                     done=torch.empty(B, dtype=torch.uint8, device=device),
                     isw=torch.empty(B, device=device))
            o["batch"] = edp.make_batch(o["obs"], o["nxt"], o["act"], o["rew"],
                                        o["done"], q=o["q"], isw=o["isw"], beta=BETA)
            self.outs.append(o)
        self.td_rounds = 64
        self.td = torch.stack([dev(fx.td_errors(self.seed, B, r), device)
                               for r in range(self.td_rounds)])
        self._init_overlap(device, self.R)
        # index sets for the kernel's back-to-back timing: a fresh sample for
        # each launch (64 sets, ~18 MB of distinct frames each), so that no
        # launch finds an earlier launch's frames in L2
        self.fresh = []
        for k in range(64):
            idx = torch.empty(B, dtype=torch.int64, device=device)
            q = torch.empty(B, dtype=torch.int32, device=device)
            edp.edp_sample(ctx, edp.EDP_SAMPLE_PRIORITIZED, B, self.seed + 1, k, idx, q)
            o = self.outs[k % self.R]
            self.fresh.append((idx, q, edp.make_batch(o["obs"], o["nxt"], o["act"], o["rew"],
                                                      o["done"], q=q, isw=o["isw"], beta=BETA)))

    def _sample(self, r, o):
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PRIORITIZED, self.B,
                            self.seed, r, o["idx"], o["q"])

    def round(self, r):
        o = self.outs[r % self.R]
        self._sample(r, o)
        self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"])
        self.edp.edp_update_priorities_td(self.ring.ctx, o["idx"],
                                          self.td[r % self.td_rounds], self.B,
                                          ALPHA, EPS)

    def round_overlap(self, r):
        """The round with the delivery on a side stream.  Delivery depends
        only on this round's sampling, so it overlaps the priority update
        (whose TD errors do not depend on the delivered batch here) and the
        next round's sampling on the main stream: the overlapped timing of
        the paper's scheduling (Sec. 6.1).  Every data dependency is kept:
        delivery r waits for sampling r; sampling r+1 follows update r in
        stream order, so it sees the updated priorities; the R output sets
        rotate, and sampling r+R waits until delivery r has read the indices
        it would overwrite."""
        k = r % self.R
        o = self.outs[k]
        self._overlapped(
            k, lambda: self._sample(r, o),
            lambda st: self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B,
                                            o["batch"], stream=st),
            lambda: self.edp.edp_update_priorities_td(
                self.ring.ctx, o["idx"], self.td[r % self.td_rounds], self.B,
                ALPHA, EPS))

    def schedules(self):
        return [("overlapped", self.round_overlap,
                 "delivery on side streams, overlapping update r and sampling r+1"),
                ("serial", self.round, "sample -> deliver -> update, one stream")]

    def deliver_once(self, r):
        idx, _, batch = self.fresh[r % len(self.fresh)]
        self.edp.edp_deliver(self.ring.ctx, idx, self.B, batch)

    def extra(self, device, mk, stream, deliver_us):
        """Ingestion (row a1) on this ring, timed after everything else: 4,096
        new transitions per call from device staging -- frames, metadata
        and their PER leaves at the running maximum priority (the deferred
        newest leaf included) with the tree above them refreshed."""
        import torch
        from paper_2609_24456_gb300 import fixtures as fx
        n = 4096
        st = torch.empty((n, self.F), dtype=torch.uint8, device=device)
        fx.content_fill_torch(self.seed, self.cap, st)
        _, action, reward, done = fx.dqn_transitions(self.seed + 1, n, with_frames=False)
        a, rw, d = dev(action, device), dev(reward, device), dev(done, device)
        us = self.time_calls(lambda: self.edp.edp_ingest(
            self.ring.ctx, st, n, action=a, reward=rw, done=d), 50, mk, stream)
        nbytes = n * (2 * self.F + 2 * 9) + n * 4
        return {"ingest": {"rows": n, "us": us, "GBs": nbytes / (us / 1e6) / 1e9,
                           "bytes_per_call": nbytes,
                           "what": "frames read + written, action/reward/done read + "
                                   "written, PER leaves written; tree refresh"}}

    def latency_step(self, r, ev_end):
        o = self.outs[r % self.R]
        self._sample(r, o)
        self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"])
        ev_end.record()
        self.edp.edp_update_priorities_td(self.ring.ctx, o["idx"],
                                          self.td[r % self.td_rounds], self.B,
                                          ALPHA, EPS)

    def e2e_setup(self, device):
        import torch
        B, K, F = self.B, self.K, self.F
        pin = lambda *s, dt=torch.float32: torch.empty(s, dtype=dt, pin_memory=True)
        self.h_td = pin(self.td_rounds, B)
        self.h_td.copy_(self.td.cpu())
        # one page-locked host batch per rotating output set; the batch's
        # outputs are these host buffers, q stays on the device (the
        # sampler's)
        self.h_outs = [dict(obs=pin(B, K, F), nxt=pin(B, K, F),
                            act=pin(B, dt=torch.int32), rew=pin(B),
                            done=pin(B, dt=torch.uint8), isw=pin(B),
                            idx=pin(B, dt=torch.int64)) for _ in range(self.R)]
        self.h_batches = [self.edp.make_batch(h["obs"], h["nxt"], h["act"], h["rew"],
                                              h["done"], q=o["q"], isw=h["isw"], beta=BETA)
                          for h, o in zip(self.h_outs, self.outs)]
        self.d_td = torch.empty(B, device=device)
        self.h2d = B * 4
        self.d2h = sum(t.numel() * t.element_size() for t in self.h_outs[0].values())

    def e2e_round(self, r):
        """User path with host buffers, in the main schedule: TD errors in,
        and each round's learner batch delivered by the kernel straight into
        a page-locked host batch on a side stream while the update and the
        next sampling run (the indices follow with a copy)."""
        k = r % self.R
        o, h = self.outs[k], self.h_outs[k]

        def deliver(st):
            self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, self.h_batches[k], stream=st)
            h["idx"].copy_(o["idx"], non_blocking=True)

        self.d_td.copy_(self.h_td[r % self.td_rounds], non_blocking=True)
        self._overlapped(
            k, lambda: self._sample(r, o), deliver,
            lambda: self.edp.edp_update_priorities_td(
                self.ring.ctx, o["idx"], self.d_td, self.B, ALPHA, EPS))

    def cpu_setup(self, host_frames=262_144):
        import numpy as np
        import oracle as orc
        from paper_2609_24456_gb300 import fixtures as fx
        self.orc = orc
        self.hcap = min(host_frames, self.cap)
        rng = np.random.default_rng(self.seed)
        self.h_frames = rng.integers(0, 256, size=(self.hcap, self.F), dtype=np.uint8)
        _, a, rw, d = fx.dqn_transitions(self.seed, self.hcap, with_frames=False)
        self.h_act, self.h_rew, self.h_done = a, rw, d
        self.st = orc.PerState(self.cap, True)
        q = orc.priorities_from_td(fx.td_errors(self.seed, self.cap), ALPHA, EPS)
        orc.ingest_leaves(self.st, 0, q)
        self.h_tds = [fx.td_errors(self.seed, self.B, r) for r in range(8)]
        self.cpu_sample = ("per-round work of this workload (B=%d stratified PER over "
                           "%d leaves, K=%d fp32 stacks + next_obs, IS weights, "
                           "priority update) reading a %d-frame host ring (%.2f GB)"
                           % (self.B, self.cap, self.K, self.hcap,
                              self.hcap * self.F / 1e9))

    def cpu_round(self, r):
        orc = self.orc
        idx, q = orc.sample_prioritized_bisect(self.st.leaves, self.B, self.seed, r)
        orc.is_weights(q, BETA)
        slots = idx % self.hcap
        orc.deliver_dqn(self.h_frames, self.h_done, self.h_act, self.h_rew,
                        self.hcap, self.hcap, self.K, slots)
        qn = orc.priorities_from_td(self.h_tds[r % 8], ALPHA, EPS)
        orc.update_leaves(self.st, self.cap, idx, qn)


class DqnTiny(Workload):
    """Uniform replay: 10,000 uint8 84x84 frames filled past capacity,
    batch 32, frame stack 4, obs + next_obs fp32; step = sample, deliver.
    Launch-bound: its headline is the sample -> batch latency."""
    name = "dqn-uniform-10k-84x84-B32"
    kernel = "k_deliver_stack"
    dtype = "u8->f32"
    launches_per_round = 2
    launches_by_schedule = {"fused": 1}

    def __init__(self, capacity=10_000, batch=32, K=4, seed=1234, out_sets=32):
        self.cap, self.B, self.K, self.seed, self.R = capacity, batch, K, seed, out_sets
        self.F = 84 * 84
        self.deliver_bytes = _stack_bytes(batch, K, self.F)
        self.round_bytes = self.deliver_bytes + batch * 8

    def config(self):
        return {"workload": self.name, "capacity": self.cap, "batch": self.B,
                "frame": "uint8 84x84", "frame_stack": self.K,
                "l2": "ring 70 MB and outputs (%d sets, %.0f MB) rotate through L2"
                      % (self.R, self.R * self.B * 2 * self.K * self.F * 4 / 1e6)}

    def setup(self, device):
        import torch
        from paper_2609_24456_gb300 import edp
        from paper_2609_24456_gb300 import fixtures as fx
        self.edp = edp
        cfg = edp.make_config(self.cap, (1, 84, 84), edp.EDP_XFORM_STACK_F32,
                              frame_stack=self.K, next_obs=True,
                              device=device.index or 0)
        self.ring = edp.Ring(cfg, reward=True)
        n = self.cap + 2345
        frames, action, reward, done = fx.dqn_transitions(self.seed, n)
        for lo in range(0, n, 4096):
            hi = min(n, lo + 4096)
            edp.edp_ingest(self.ring.ctx, dev(frames[lo:hi], device), hi - lo,
                           action=dev(action[lo:hi], device),
                           reward=dev(reward[lo:hi], device),
                           done=dev(done[lo:hi], device))
        edp.edp_sync(self.ring.ctx)
        self.host = (frames, action, reward, done, n)
        B, K, F = self.B, self.K, self.F
        self.outs = []
        for _ in range(self.R):
            o = dict(idx=torch.empty(B, dtype=torch.int64, device=device),
                     obs=torch.empty((B, K, F), device=device),
                     nxt=torch.empty((B, K, F), device=device),
                     act=torch.empty(B, dtype=torch.int32, device=device),
                     rew=torch.empty(B, device=device),
                     done=torch.empty(B, dtype=torch.uint8, device=device))
            o["batch"] = edp.make_batch(o["obs"], o["nxt"], o["act"], o["rew"], o["done"])
            self.outs.append(o)

    def round(self, r):
        o = self.outs[r % self.R]
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_UNIFORM, self.B,
                            self.seed, r, o["idx"])
        self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"])

    def round_fused(self, r):
        o = self.outs[r % self.R]
        self.edp.edp_sample_deliver(self.ring.ctx, self.B, self.seed, r, o["idx"], o["batch"])

    def schedules(self):
        return [("fused", self.round_fused, "uniform draw inside the delivery kernel "
                 "(edp_sample_deliver), one launch per batch"),
                ("sample+deliver", self.round, "edp_sample then edp_deliver, one stream")]

    def deliver_once(self, r):
        o = self.outs[r % self.R]
        self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"])

    def latency_step(self, r, ev_end):
        self.round_fused(r)
        ev_end.record()

    def e2e_setup(self, device):
        import torch
        B, K, F = self.B, self.K, self.F
        pin = lambda *s, dt=torch.float32: torch.empty(s, dtype=dt, pin_memory=True)
        self.h_out = dict(obs=pin(B, K, F), nxt=pin(B, K, F),
                          act=pin(B, dt=torch.int32), rew=pin(B),
                          done=pin(B, dt=torch.uint8), idx=pin(B, dt=torch.int64))
        self.h2d = 0
        self.d2h = sum(t.numel() * t.element_size() for t in self.h_out.values())
        self.h_outs = [self.h_out] + [{k: torch.empty_like(t, pin_memory=True)
                                       for k, t in self.h_out.items()}]
        self.h_batches = [self.edp.make_batch(h["obs"], h["nxt"], h["act"], h["rew"],
                                              h["done"]) for h in self.h_outs]
        self.sides = [torch.cuda.Stream(device=device) for _ in range(2)]

    def e2e_round(self, r):
        """The main schedule's call with host buffers: the kernel draws the
        batch and writes it straight into a page-locked host batch, the
        calls alternating between two side streams (each writes its own host
        batch, so stream order protects its reuse) so consecutive batches
        overlap; the indices (device) follow with a copy."""
        import torch
        k = r % 2
        o, side = self.outs[k], self.sides[k]
        if not getattr(self, "side_used", False):
            fork = torch.cuda.Event()
            fork.record()
            for st in self.sides:
                st.wait_event(fork)
        self.side_used = True
        with torch.cuda.stream(side):
            self.edp.edp_sample_deliver(self.ring.ctx, self.B, self.seed, r, o["idx"],
                                        self.h_batches[k], stream=side)
            self.h_outs[k]["idx"].copy_(o["idx"], non_blocking=True)

    def cpu_setup(self):
        import numpy as np
        import oracle as orc
        from paper_2609_24456_gb300 import fixtures as fx
        self.orc = orc
        if not hasattr(self, "host"):
            n = self.cap + 2345
            self.host = fx.dqn_transitions(self.seed, n) + (n,)
        frames, action, reward, done, n = self.host
        self.h_frames = np.zeros((self.cap, self.F), np.uint8)
        self.h_act = np.zeros(self.cap, np.int32)
        self.h_rew = np.zeros(self.cap, np.float32)
        self.h_done = np.zeros(self.cap, np.uint8)
        for arr, src in [(self.h_frames, frames), (self.h_act, action),
                         (self.h_rew, reward), (self.h_done, done)]:
            orc.ring_write(arr, self.cap, 0, np.ascontiguousarray(src))
        self.total = n
        self.cpu_sample = "rounds of this workload on the full 10,000-frame host ring"

    def cpu_round(self, r):
        idx = self.orc.sample_uniform(self.cap, self.total, self.cap - 1, self.B,
                                      self.seed, r)
        self.orc.deliver_dqn(self.h_frames, self.h_done, self.h_act, self.h_rew,
                             self.cap, self.total, self.K, idx)


class PpoIteration(Workload):
    """On-policy iteration: 256 envs x 128 steps of uint8 64x64x3 obs; GAE
    (gamma 0.99, lambda 0.95) with global advantage normalisation, Philox
    shuffle of 32,768 samples into 8 mini-batches of 4,096, each delivered as
    bf16 [4096,3,64,64] with gathered advantages and returns.  Step = one
    iteration (GAE + shuffle + 8 deliveries); the rollout ingest is timed
    separately."""
    name = "ppo-iteration-256x128-64x64x3"
    kernel = "k_deliver_hwc"
    dtype = "u8->bf16,f64"
    T, E, H, W, C, M = 128, 256, 64, 64, 3, 8

    def __init__(self, seed=1236, sched=True):
        self.seed, self.sched = seed, sched
        self.n = self.T * self.E
        self.mb = self.n // self.M
        F = self.H * self.W * self.C
        self.F = F
        # per delivered sample: obs read + bf16 write + adv/ret gathers + idx
        self.sample_bytes = F + 2 * F + 8 + 8 + 8
        # the main schedule delivers the whole iteration in one call
        self.deliver_bytes = self.n * self.sample_bytes
        gae = self.T * self.E * (4 + 1 + 4) + self.E * 4 + 3 * self.T * self.E * 4
        perm = self.n * (8 + 8 + 8 + 4 + 8 + 4 + 8) + 3 * 4 * (self.n // 4)
        self.round_bytes = gae + perm + self.n * self.sample_bytes
        self.launches_per_round = 2 + 3 + 1  # GAE, shuffle, delivery

    def config(self):
        return {"workload": self.name, "envs": self.E, "steps": self.T,
                "obs": "uint8 64x64x3 HWC -> bf16 CHW", "minibatches": self.M,
                "gamma": 0.99, "lambda": 0.95,
                "l2": "rollout 403 MB > L2; mini-batch outputs 805 MB per iteration"}

    def setup(self, device):
        import torch
        from paper_2609_24456_gb300 import edp
        from paper_2609_24456_gb300 import fixtures as fx
        self.edp = edp
        cfg = edp.make_config(self.n, (self.C, self.H, self.W),
                              edp.EDP_XFORM_HWC_CHW_BF16, device=device.index or 0)
        self.ring = edp.Ring(cfg, action=False, reward=False, done=False)
        obs, r, v, d = fx.ppo_rollout(self.seed, self.T, self.E)
        self.h_obs, self.h_r, self.h_v, self.h_d = obs, r, v, d
        self.d_obs = dev(obs, device)
        self.r, self.v, self.d = dev(r, device), dev(v, device), dev(d, device)
        edp.edp_ingest(self.ring.ctx, self.d_obs, self.n)
        T, E = self.T, self.E
        self.adv = torch.empty((T, E), device=device)
        self.ret = torch.empty((T, E), device=device)
        self.nrm = torch.empty((T, E), device=device)
        self.idx = torch.empty(self.n, dtype=torch.int64, device=device)
        self.out = [torch.empty((self.mb, self.C, self.H, self.W), dtype=torch.bfloat16,
                                device=device) for _ in range(2)]
        self.a_out = torch.empty(self.mb, device=device)
        self.r_out = torch.empty(self.mb, device=device)
        # all M mini-batches of one iteration, mini-batch m = rows
        # [m * 4096, (m + 1) * 4096) (805 MB, larger than L2)
        self.out_all = torch.empty((self.n, self.C, self.H, self.W), dtype=torch.bfloat16,
                                   device=device)
        self.a_all = torch.empty(self.n, device=device)
        self.r_all = torch.empty(self.n, device=device)
        self.side = torch.cuda.Stream(device=device)
        self.sides = [self.side]
        self.fork = torch.cuda.Event()
        self.gae_done = torch.cuda.Event()
        # first calls allocate scratch outside any capture
        self._gae()
        edp.edp_sample(self.ring.ctx, edp.EDP_SAMPLE_PERMUTE, self.n, self.seed, 0, self.idx)
        edp.edp_sync(self.ring.ctx)

    def _gae(self):
        self.edp.edp_gae(self.ring.ctx, self.r, self.v, self.d, self.T, self.E,
                         0.99, 0.95, self.adv, self.ret, self.nrm)

    def _mb(self, m, r):
        sub = self.idx[m * self.mb:(m + 1) * self.mb]
        b = self.edp.make_batch(self.out[(r * self.M + m) % 2],
                                gather=[(self.nrm.view(-1), self.a_out),
                                        (self.ret.view(-1), self.r_out)])
        self.edp.edp_deliver(self.ring.ctx, sub, self.mb, b)

    def round(self, r):
        self._gae()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        for m in range(self.M):
            self._mb(m, r)

    def _deliver_all(self, parts=1):
        """The iteration's deliveries in `parts` calls (granularity
        g_del = 1 / parts); call p fills rows [p n / parts, (p+1) n / parts)
        of the output."""
        m = self.n // parts
        for p in range(parts):
            sl = slice(p * m, (p + 1) * m)
            b = self.edp.make_batch(self.out_all[sl],
                                    gather=[(self.nrm.view(-1), self.a_all[sl]),
                                            (self.ret.view(-1), self.r_all[sl])])
            self.edp.edp_deliver(self.ring.ctx, self.idx[sl], m, b)

    def round_parts(self, r, parts):
        """GAE on a side stream beside the shuffle (the two are independent:
        GAE reads the rollout scalars, the shuffle only its keys), then the
        iteration's delivery in `parts` calls: delivery granularity
        g_del = 1 / parts (Sec. 4.2).  With parts = 1 a single call delivers
        all mini-batches; mini-batch m is rows [4096 m, 4096 (m + 1)) of the
        output, equal to what the m-th per-mini-batch call delivers."""
        import torch
        main = torch.cuda.current_stream()
        self.fork.record()  # the side stream starts after prior work
        self.side_used = True
        with torch.cuda.stream(self.side):
            self.side.wait_event(self.fork)
            self.edp.edp_gae(self.ring.ctx, self.r, self.v, self.d, self.T, self.E,
                             0.99, 0.95, self.adv, self.ret, self.nrm, stream=self.side)
            self.gae_done.record()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        main.wait_event(self.gae_done)
        self._deliver_all(parts)

    def round_batched(self, r):
        self.round_parts(r, 1)

    def schedules(self):
        """The delivery-granularity sweep of Sec. 6.1 on this iteration:
        g_del = 1 (main), 1/2, 1/4 and 1/8 with GAE beside the shuffle, and
        the plain one-stream iteration with one call per mini-batch."""
        sweep = [("g=1/%d" % k, (lambda r, k=k: self.round_parts(r, k)),
                  "GAE on a side stream beside the shuffle; %d delivery calls of "
                  "%d samples (g_del = 1/%d)" % (k, self.n // k, k)) for k in (2, 4, 8)]
        return [("batched", self.round_batched,
                 "GAE on a side stream beside the shuffle; one delivery call "
                 "for all 8 mini-batches (g_del = 1)")] + sweep + [
                ("per-minibatch", self.round,
                 "GAE, shuffle, 8 mini-batch deliveries of 4,096, one stream "
                 "(g_del = 1/8)")]

    def deliver_once(self, r):
        self._deliver_all()

    def extra(self, device, mk, stream, deliver_us):
        """Rollout ingestion (row a1), reported beside the iteration as the
        workload asks: the 32,768 observations of a rollout copied from the
        actors' device buffer into the ring (402.7 MB read + 402.7 MB
        written)."""
        us = self.time_calls(lambda: self.edp.edp_ingest(self.ring.ctx, self.d_obs, self.n),
                             50, mk, stream)
        nbytes = 2 * self.n * self.F
        out = {"ingest": {"rows": self.n, "us": us, "GBs": nbytes / (us / 1e6) / 1e9,
                          "bytes_per_call": nbytes,
                          "what": "rollout observations device -> ring"}}
        if self.sched:
            out["sched"] = self.sched_experiment(device, mk, stream)
        return out

    # -- latency-aware scheduling, measured (Sec. 6; the auto-versus-manual
    # comparison of Sec. 7, reproduced with synthetic data) ----------------
    def _learn(self, m):
        """Stand-in learner update on mini-batch m: one bf16 GEMM over its
        observations (4,096 x 12,288 @ 12,288 x 512, cuBLAS), about the cost
        of a small policy network's forward and backward pass."""
        import torch
        x = self.out_all[m * self.mb:(m + 1) * self.mb].view(self.mb, -1)
        torch.matmul(x, self.w_learn, out=self.y_learn)

    def _iteration(self, r, parts, overlap):
        """Ingest the rollout, GAE beside the shuffle, then the delivery in
        `parts` calls and the learner on every mini-batch: inline (deliver
        part c, learn its mini-batches, next part), or overlapped (the parts
        delivered on a side stream back to back, the learner on part c once
        its delivery has finished: mini-batch pipelining)."""
        import torch
        main = torch.cuda.current_stream()
        self.edp.edp_ingest(self.ring.ctx, self.d_obs, self.n)
        self.fork.record()
        with torch.cuda.stream(self.side):
            self.side.wait_event(self.fork)
            self.edp.edp_gae(self.ring.ctx, self.r, self.v, self.d, self.T, self.E,
                             0.99, 0.95, self.adv, self.ret, self.nrm, stream=self.side)
            self.gae_done.record()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        main.wait_event(self.gae_done)
        m_per = self.M // parts
        rows = self.n // parts

        def deliver(c, st=None):
            sl = slice(c * rows, (c + 1) * rows)
            b = self.edp.make_batch(self.out_all[sl],
                                    gather=[(self.nrm.view(-1), self.a_all[sl]),
                                            (self.ret.view(-1), self.r_all[sl])])
            self.edp.edp_deliver(self.ring.ctx, self.idx[sl], rows, b, stream=st)

        if not overlap:
            for c in range(parts):
                deliver(c)
                for m in range(c * m_per, (c + 1) * m_per):
                    self._learn(m)
            return
        self.fork.record()
        with torch.cuda.stream(self.side):
            self.side.wait_event(self.fork)
            for c in range(parts):
                deliver(c, self.side)
                self.part_done[c].record()
        for c in range(parts):
            main.wait_event(self.part_done[c])
            for m in range(c * m_per, (c + 1) * m_per):
                self._learn(m)
        main.wait_stream(self.side)

    def sched_experiment(self, device, mk, stream, reps=20):
        """Profile the operator costs once, let edp_sched_choose pick the
        delivery timing and granularity (Eq. 2), and time every feasible
        configuration to see whether the pick is the fastest.  On-policy
        candidates: g_del = k/8 for k | 8.  Overlap means pipelining within
        the iteration, so it needs g_del < 1; g_del = 1 runs inline only."""
        import torch
        self.w_learn = torch.randn(self.F, 512, device=device).to(torch.bfloat16) * 0.01
        self.y_learn = torch.empty(self.mb, 512, device=device, dtype=torch.bfloat16)
        self.part_done = [torch.cuda.Event() for _ in range(self.M)]
        G = self.edp.edp_sched_granularities(True, self.M)
        # profiled costs (us): learner update of one iteration, one delivery
        # invocation at each g, the ingestion side (ingest + GAE beside the
        # shuffle), and one cross-stream hand-off
        t_update = self.time_calls(lambda: [self._learn(m) for m in range(self.M)],
                                   reps, mk, stream)
        t_del = []
        for g in G:
            rows = int(round(g * self.n))
            sl = slice(0, rows)
            b = self.edp.make_batch(self.out_all[sl],
                                    gather=[(self.nrm.view(-1), self.a_all[sl]),
                                            (self.ret.view(-1), self.r_all[sl])])
            t_del.append(self.time_calls(
                lambda: self.edp.edp_deliver(self.ring.ctx, self.idx[sl], rows, b),
                reps, mk, stream))

        def ing_side():
            self.edp.edp_ingest(self.ring.ctx, self.d_obs, self.n)
            self.fork.record()
            with torch.cuda.stream(self.side):
                self.side.wait_event(self.fork)
                self.edp.edp_gae(self.ring.ctx, self.r, self.v, self.d, self.T, self.E,
                                 0.99, 0.95, self.adv, self.ret, self.nrm,
                                 stream=self.side)
                self.gae_done.record()
            self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                                self.seed, 0, self.idx)
            torch.cuda.current_stream().wait_event(self.gae_done)
        t_ing = self.time_calls(ing_side, reps, mk, stream)

        def handoff():
            self.fork.record()
            with torch.cuda.stream(self.side):
                self.side.wait_event(self.fork)
                self.y_learn[:1, :1].zero_()
                self.gae_done.record()
            torch.cuda.current_stream().wait_event(self.gae_done)
        t_sync = self.time_calls(handoff, reps, mk, stream)
        nd = len(G)
        feasible = [(o, j) for o in (0, 1) for j in range(nd) if not (o and G[j] >= 1)]

        def pick(c_del):
            _, scores = self.edp.edp_sched_choose(0.0, t_update, 0.0, t_sync, [1.0], [t_ing],
                                                  G, t_del, all_scores=True,
                                                  contention_del=c_del)
            pred = {(o, j): scores[o * nd + j] for (o, j) in feasible}  # o_ing = 0
            return min(feasible, key=lambda k: (pred[k], k)), pred

        measured = {(o, j): self.time_calls(
            lambda: self._iteration(0, int(round(1 / G[j])), o), reps, mk, stream)
            for (o, j) in feasible}
        fastest = min(measured, key=measured.get)
        paper_pick, paper_pred = pick(0.0)
        # one probe pair calibrates the contention: inline and overlapped at
        # the finest granularity; the share of the model's hidden time that
        # the overlap actually saved
        j0 = 0
        tbar = t_del[j0] / G[j0]
        hide0 = (1.0 - G[j0]) * min(t_update, tbar)
        saved = measured[(0, j0)] - measured[(1, j0)] + t_sync
        c_del = min(1.0, max(0.0, 1.0 - saved / hide0)) if hide0 > 0 else 1.0
        cal_pick, cal_pred = pick(c_del)
        fmt = lambda k: {"g_del": G[k[1]], "overlap_del": k[0]}
        return {"costs_us": {"t_update": t_update, "t_ing": t_ing, "t_sync_del": t_sync,
                             "t_del": dict(zip(["%g" % g for g in G], t_del))},
                "configs": [dict(fmt(k), measured_us=measured[k],
                                 predicted_us=paper_pred[k],
                                 predicted_calibrated_us=cal_pred[k]) for k in feasible],
                "fastest": fmt(fastest),
                "paper_model": dict(fmt(paper_pick),
                                    over_fastest=measured[paper_pick] / measured[fastest]),
                "calibrated": dict(fmt(cal_pick), contention_del=c_del,
                                   over_fastest=measured[cal_pick] / measured[fastest])}

    def latency_step(self, r, ev_end):
        self._gae()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        self._mb(0, r)
        ev_end.record()

    def e2e_setup(self, device):
        import torch
        pin = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        self.h_in = [pin(t) for t in (self.r, self.v, self.d)]
        for h, t in zip(self.h_in, (self.r, self.v, self.d)):
            h.copy_(t.cpu())
        # all 8 mini-batches of an iteration, mini-batch m = rows
        # [4096 m, 4096 (m + 1)), written by the delivery straight into
        # page-locked host memory
        self.h_all = pin(self.out_all)
        self.h_aall = pin(self.a_all)
        self.h_rall = pin(self.r_all)
        self.h2d = sum(t.numel() * t.element_size() for t in self.h_in)
        self.d2h = self.h_all.numel() * 2 + 8 * self.n
        self.h_batch = self.edp.make_batch(self.h_all,
                                           gather=[(self.nrm.view(-1), self.h_aall),
                                                   (self.ret.view(-1), self.h_rall)])

    def e2e_round(self, r):
        """One stream: the rollout's scalars in, GAE, shuffle, and the
        iteration's delivery (one call) written straight into the page-locked
        host batch."""
        for h, t in zip(self.h_in, (self.r, self.v, self.d)):
            t.copy_(h, non_blocking=True)
        self._gae()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        self.edp.edp_deliver(self.ring.ctx, self.idx, self.n, self.h_batch)

    def cpu_setup(self):
        import oracle as orc
        from paper_2609_24456_gb300 import fixtures as fx
        self.orc = orc
        if not hasattr(self, "h_obs"):
            self.h_obs, self.h_r, self.h_v, self.h_d = fx.ppo_rollout(
                self.seed, self.T, self.E)
        self.cpu_sample = "whole iterations of this workload (GAE direct sums, shuffle, 8 mini-batches)"

    def cpu_round(self, r):
        import numpy as np
        orc = self.orc
        adv, ret = orc.gae(self.h_r, self.h_v, self.h_d, 0.99, 0.95)
        nrm, _, _ = orc.normalize(adv.ravel())
        perm = orc.permutation(self.n, self.seed, r)
        nrm32, ret32 = nrm.astype(np.float32), ret.ravel().astype(np.float32)
        for m in range(self.M):
            orc.deliver_ppo(self.h_obs, self.n, self.n, self.H, self.W, self.C,
                            perm[m * self.mb:(m + 1) * self.mb], nrm32, ret32)


MEAN3, STD3 = (0.485, 0.456, 0.406), (0.229, 0.224, 0.225)


class MmReplay(Workload):
    """Multimodal replay: 200,000 transitions of uint8 3x224x224 images
    (~30.1 GB) + 512 int32 tokens + reward, uniform batch 1,024 delivered as
    per-channel normalised bf16 with collated tokens and rewards; step =
    sample, deliver.  With hbm_frac < 1 the oldest part of the ring lives in
    page-locked host memory (two-tier placement) and each step also ingests
    4,096 new transitions from page-locked staging, demoting the oldest HBM
    entries."""
    kernel = "k_deliver_norm"
    dtype = "u8->bf16"
    C, H, W, L = 3, 224, 224, 512

    def __init__(self, capacity=200_000, batch=1024, seed=1237, hbm_frac=1.0,
                 ingest=0):
        self.cap, self.B, self.seed = capacity, batch, seed
        self.cap_h = int(capacity * hbm_frac)
        self.ingest = ingest
        self.F = self.C * self.H * self.W
        self.tiered = self.cap_h < self.cap
        self.name = ("mm-tiered-%dk-%dk-host-B%d" % (self.cap // 1000,
                                                    (self.cap - self.cap_h) // 1000, batch)
                     if self.tiered else "mm-replay-%dk-3x224x224-B%d" % (capacity // 1000, batch))
        per = self.F + 4 * self.L + 4  # bytes read per sample
        self.deliver_bytes = batch * (per + 2 * self.F + 4 * self.L + 4 + 8)
        rec = self.F + 4 * self.L + 4
        self.ingest_bytes = ingest * (2 * rec + 4)  # staging read + HBM write
        self.demote_bytes = ingest * 2 * (self.F + 4 * self.L)
        self.round_bytes = self.deliver_bytes + batch * 8 + self.ingest_bytes + \
            (self.demote_bytes if self.tiered else 0)
        self.launches_per_round = 2 + (3 if ingest else 0)  # + swap obs, swap tokens, metadata
        self.launches_by_schedule = {"fused overlapped": 1}  # one fused launch per step

    def split_bytes(self):
        """Per-step bytes by where they move (two-tier only): over HBM, and
        over the host link in each direction."""
        if not self.tiered:
            return None
        row = self.F + 4 * self.L
        host_frac = (self.cap - self.cap_h) / self.cap
        host_reads = self.B * host_frac * row
        return {"hbm": (2 * self.ingest * row + self.B * (1 - host_frac) * row
                        + self.B * (2 * self.F + 4 * self.L + 4 + 8)),
                "link_in": self.ingest * row + host_reads,
                "link_out": self.ingest * row}

    def config(self):
        c = {"workload": self.name, "capacity": self.cap, "batch": self.B,
             "obs": "uint8 3x224x224 CHW -> bf16 normalised", "tokens": self.L,
             "resident_hbm_GB": round(self.cap_h * (self.F + 4 * self.L) / 1e9, 1)}
        if self.tiered:
            c.update({"host_tier": self.cap - self.cap_h, "ingest_per_step": self.ingest,
                      "host_GB": round((self.cap - self.cap_h) * (self.F + 4 * self.L) / 1e9, 1)})
        return c

    def setup(self, device):
        import torch
        from paper_2609_24456_gb300 import edp
        from paper_2609_24456_gb300 import fixtures as fx
        self.edp = edp
        cfg = edp.make_config(self.cap, (self.C, self.H, self.W),
                              edp.EDP_XFORM_CHW_NORM_BF16, hbm_capacity=self.cap_h,
                              tokens=self.L, norm_mean=MEAN3, norm_std=STD3,
                              device=device.index or 0)
        self.ring = edp.Ring(cfg, action=False, done=False)
        _, rew = fx.mm_metadata(self.seed, self.cap + max(self.ingest, 1) * 64, tokens=0)
        self.rew_all = rew
        chunk = 4096
        obs = torch.empty((chunk, self.F), dtype=torch.uint8, device=device)
        tok = torch.empty((chunk, self.L), dtype=torch.int32, device=device)
        for lo in range(0, self.cap, chunk):
            n = min(chunk, self.cap - lo)
            fx.content_fill_torch(self.seed, lo, obs[:n])
            fx.token_fill_torch(self.seed, lo, tok[:n])
            edp.edp_ingest(self.ring.ctx, obs[:n], n, tokens=tok[:n],
                           reward=dev(rew[lo:lo + n], device))
        edp.edp_sync(self.ring.ctx)
        self.total0 = self.cap
        if self.ingest:
            # page-locked staging of new transitions (actors on the host)
            n = self.ingest
            self.st_obs = torch.empty((n, self.F), dtype=torch.uint8, pin_memory=True)
            self.st_tok = torch.empty((n, self.L), dtype=torch.int32, pin_memory=True)
            fx.content_fill_torch(self.seed, self.cap, obs[:n])
            fx.token_fill_torch(self.seed, self.cap, tok[:n])
            self.st_obs.copy_(obs[:n])
            self.st_tok.copy_(tok[:n])
            self.st_rew = torch.from_numpy(rew[:n].copy()).pin_memory()
        del obs, tok
        B = self.B
        self.outs = []
        for _ in range(2):
            o = dict(idx=torch.empty(B, dtype=torch.int64, device=device),
                     obs=torch.empty((B, self.C, self.H, self.W), dtype=torch.bfloat16,
                                     device=device),
                     tok=torch.empty((B, self.L), dtype=torch.int32, device=device),
                     rew=torch.empty(B, device=device))
            o["batch"] = edp.make_batch(o["obs"], tokens=o["tok"], reward=o["rew"])
            self.outs.append(o)
        self._init_overlap(device, len(self.outs))

    def round(self, r):
        ctx = self.ring.ctx
        if self.ingest:
            self.edp.edp_ingest(ctx, self.st_obs, self.ingest, tokens=self.st_tok,
                                reward=self.st_rew)
        o = self.outs[r % 2]
        self.edp.edp_sample(ctx, self.edp.EDP_SAMPLE_UNIFORM, self.B, self.seed, r, o["idx"])
        self.edp.edp_deliver(ctx, o["idx"], self.B, o["batch"])

    def round_overlap(self, r):
        """Delivery r on a side stream while round r+1 samples (no ingest:
        an ingest would overwrite rows a pending delivery reads)."""
        k = r % 2
        o = self.outs[k]
        self._overlapped(
            k, lambda: self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_UNIFORM,
                                           self.B, self.seed, r, o["idx"]),
            lambda st: self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"],
                                            stream=st))

    def round_fused(self, r):
        """Fused sample -> deliver calls alternating between two side
        streams: output set k is always written from side stream k, so
        stream order protects its reuse; consecutive batches overlap."""
        import torch
        k = r % 2
        o = self.outs[k]
        side = self.sides[k]
        if not self.side_used:
            self.fork_ev = torch.cuda.Event()
            self.fork_ev.record()
            for st in self.sides:
                st.wait_event(self.fork_ev)
        self.side_used = True
        with torch.cuda.stream(side):
            self.edp.edp_sample_deliver(self.ring.ctx, self.B, self.seed, r, o["idx"],
                                        o["batch"], stream=side)

    def schedules(self):
        one = ("one stream", self.round, "sample -> deliver, one stream")
        if self.ingest:
            return [one]
        return [("fused overlapped", self.round_fused,
                 "uniform draw inside the delivery kernel (edp_sample_deliver), "
                 "calls alternating between two side streams"),
                ("overlapped", self.round_overlap,
                 "delivery on side streams, overlapping sampling r+1"), one]

    def deliver_once(self, r):
        o = self.outs[r % 2]
        self.edp.edp_deliver(self.ring.ctx, o["idx"], self.B, o["batch"])

    def latency_step(self, r, ev_end):
        o = self.outs[r % 2]
        self.edp.edp_sample_deliver(self.ring.ctx, self.B, self.seed, r, o["idx"], o["batch"])
        ev_end.record()

    def e2e_setup(self, device):
        import torch
        o = self.outs[0]
        self.h_out = {k: torch.empty(o[k].shape, dtype=o[k].dtype, pin_memory=True)
                      for k in ("obs", "tok", "rew", "idx")}
        self.h2d = 0 if not self.ingest else self.ingest * (self.F + 4 * self.L + 4)
        self.d2h = sum(t.numel() * t.element_size() for t in self.h_out.values())
        h = self.h_out
        self.h_batch = self.edp.make_batch(h["obs"], tokens=h["tok"], reward=h["rew"])

    def e2e_round(self, r):
        """One stream: (ingest,) sample, and the delivery written straight
        into the page-locked host batch; the indices follow with a copy."""
        ctx = self.ring.ctx
        if self.ingest:
            self.edp.edp_ingest(ctx, self.st_obs, self.ingest, tokens=self.st_tok,
                                reward=self.st_rew)
        o = self.outs[0]
        self.edp.edp_sample(ctx, self.edp.EDP_SAMPLE_UNIFORM, self.B, self.seed, r, o["idx"])
        self.edp.edp_deliver(ctx, o["idx"], self.B, self.h_batch)
        self.h_out["idx"].copy_(o["idx"], non_blocking=True)

    def extra(self, device, mk, stream, deliver_us):
        """Two-tier: host-link bandwidth measured in this run (zero-copy read
        kernel and a pinned H2D copy) and the host-tier share of the
        delivery's reads against it.  Single tier: the placement experiment
        (bandwidth table, placement map, and the model checked against
        measured transfers at this workload's sample size)."""
        if not self.tiered:
            return {"placement": self.placement_experiment(device, mk, stream, deliver_us)}
        import torch
        from paper_2609_24456_gb300 import edp
        nbytes = 4 << 30
        h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
        h.fill_(3)
        d = torch.empty(nbytes, dtype=torch.uint8, device=device)
        fold = torch.zeros(1, dtype=torch.int64, device=device)
        best_probe = best_copy = 0.0
        for _ in range(3):
            e0, e1 = mk(), mk()
            e0.record(stream)
            edp.edp_probe_host_read(h, nbytes, fold)
            e1.record(stream)
            torch.cuda.synchronize()
            best_probe = max(best_probe, nbytes / (e0.elapsed_time(e1) / 1e3) / 1e9)
            e0.record(stream)
            d.copy_(h, non_blocking=True)
            e1.record(stream)
            torch.cuda.synchronize()
            best_copy = max(best_copy, nbytes / (e0.elapsed_time(e1) / 1e3) / 1e9)
        del h, d
        link = max(best_probe, best_copy)
        host_frac = (self.cap - self.cap_h) / self.cap
        host_bytes = self.B * host_frac * (self.F + 4 * self.L)
        achieved = host_bytes / (deliver_us / 1e6) / 1e9
        return {"host_link": {"probe_read_GBs": best_probe, "h2d_copy_GBs": best_copy,
                              "delivery_host_read_GBs": achieved,
                              "frac_of_link": achieved / link,
                              "host_bytes_per_delivery": host_bytes}}

    def placement_experiment(self, device, mk, stream, deliver_us, rows=16384):
        """Bandwidth-aware placement on this node (Sec. 5; the placement
        sweep of Sec. 7, reproduced with synthetic data): profile the
        effective bandwidths once (edp_place_profile), build the candidate
        placements for CPU actors and a learner on this GPU, and let the
        library solve Eq. 1 over per-sample sizes (the placement map) at the
        paper's sweep capacity of 10^6.  Then, at this workload's sample
        (150,528-byte image + 2,048 bytes of tokens), time both legs of each
        placement with the mechanism its bandwidths stand for -- CPU actors
        copying into host memory, or the GPU reading page-locked staging;
        the learner's batch gathered on the CPU and copied (pageable),
        delivered by the kernel from page-locked memory in place (pinned),
        or from HBM -- and compare the ranking."""
        import numpy as np
        import torch
        from paper_2609_24456_gb300 import edp
        from paper_2609_24456_gb300 import fixtures as fx
        bw = edp.edp_place_profile(device.index or 0, 1 << 30)
        x = self.F + 4 * self.L
        ring_bytes = self.cap * x
        mem_gpu = bw["hbm_free"] + ring_bytes - 8e9  # this ring's HBM is the buffer's
        mem_host = 0.8 * _mem_available()
        def best_of(fn, k=3):
            t = []
            for _ in range(k):
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                fn()
                torch.cuda.synchronize()
                t.append(time.perf_counter() - t0)
            return min(t)

        n_in, B = 4096, self.B
        rng = np.random.default_rng(self.seed)
        stage = torch.empty((n_in, x), dtype=torch.uint8, pin_memory=True)
        stage.numpy()[:] = rng.integers(0, 256, size=(n_in, x), dtype=np.uint8)
        sel = np.sort(rng.integers(0, rows, size=B))
        meas = {}
        # host pageable: actors memcpy into the ring; the learner's batch is
        # gathered on the CPU into page-locked staging and copied in
        page = np.empty((rows, x), dtype=np.uint8)
        page[:] = 1
        t_in = best_of(lambda: np.copyto(page[:n_in], stage.numpy())) / n_in
        pin_b = torch.empty((B, x), dtype=torch.uint8, pin_memory=True)
        dev_b = torch.empty((B, x), dtype=torch.uint8, device=device)

        def gather_copy():
            np.take(page, sel, axis=0, out=pin_b.numpy())
            dev_b.copy_(pin_b, non_blocking=True)
        t_gc = best_of(gather_copy)
        meas["host_pageable"] = t_in + t_gc / B
        del page
        # the pageable path's out-leg bandwidth is that of its mechanism, a
        # CPU gather then a pageable copy, measured here at this row size
        bw_gather_copy = B * x / t_gc
        names = ["host_pageable", "host_pinned", "gpu", "gpu+host"]
        opts = [dict(kind=edp.EDP_PLACE_HOST_PAGEABLE, bw_in=bw["host_copy"],
                     bw_out=bw_gather_copy, mem=mem_host),
                dict(kind=edp.EDP_PLACE_HOST_PINNED, bw_in=bw["host_copy"],
                     bw_out=bw["zero_copy_read"], mem=mem_host),
                dict(kind=edp.EDP_PLACE_GPU, bw_in=bw["h2d_pinned"], bw_out=bw["hbm_copy"],
                     mem=mem_gpu),
                dict(kind=edp.EDP_PLACE_GPU_HOST, bw_in=bw["h2d_pinned"],
                     bw_out=bw["hbm_copy"], mem=mem_gpu, bw_out2=bw["zero_copy_read"],
                     mem2=mem_host)]
        xs = [int(512 * 2 ** (k / 2)) for k in range(25)]  # 512 B .. 2 MiB, half octaves
        pmap = edp.edp_place_map(opts, 1e6, xs)
        best, t_pred = edp.edp_place_choose(opts, self.cap, x)


        # host pinned: actors memcpy into page-locked memory; the kernel
        # delivers from it in place (a ring whose HBM tier holds one entry)
        cfg = edp.make_config(rows, (self.C, self.H, self.W), edp.EDP_XFORM_CHW_NORM_BF16,
                              hbm_capacity=1, tokens=self.L, norm_mean=MEAN3,
                              norm_std=STD3, device=device.index or 0)
        pr = edp.Ring(cfg, action=False, reward=False, done=False)
        obs = torch.empty((n_in, self.F), dtype=torch.uint8, device=device)
        tok = torch.empty((n_in, self.L), dtype=torch.int32, device=device)
        for lo in range(0, rows, n_in):
            fx.content_fill_torch(self.seed, lo, obs)
            fx.token_fill_torch(self.seed, lo, tok)
            edp.edp_ingest(pr.ctx, obs, n_in, tokens=tok)
        hobs = pr.host_obs.numpy()
        t_in = best_of(lambda: np.copyto(hobs[:n_in], stage.numpy()[:, :self.F])) / n_in
        idx = torch.empty(B, dtype=torch.int64, device=device)
        out = self.outs[0]
        batch = edp.make_batch(out["obs"], tokens=out["tok"])
        edp.edp_sample(pr.ctx, edp.EDP_SAMPLE_UNIFORM, B, self.seed, 0, idx)
        t_out = self.time_calls(lambda: edp.edp_deliver(pr.ctx, idx, B, batch), 20, mk,
                                stream) * 1e-6
        meas["host_pinned"] = t_in + t_out / B
        pr.close()
        del pr, hobs
        # GPU: the ingest kernel reads page-locked staging into HBM; the
        # delivery kernel gathers from HBM (its time measured above)
        st_obs = torch.empty((n_in, self.F), dtype=torch.uint8, pin_memory=True)
        st_tok = torch.empty((n_in, self.L), dtype=torch.int32, pin_memory=True)
        st_rew = torch.zeros(n_in, dtype=torch.float32, pin_memory=True)
        st_obs.numpy()[:] = stage.numpy()[:, :self.F]
        st_tok.numpy()[:] = 7
        t_in = self.time_calls(lambda: edp.edp_ingest(self.ring.ctx, st_obs, n_in,
                                                      tokens=st_tok, reward=st_rew),
                               10, mk, stream) * 1e-6 / n_in
        meas["gpu"] = t_in + deliver_us * 1e-6 / B
        # the two-tier placement holds this buffer in HBM alone (h = 1): its
        # transfers are the GPU placement's
        meas["gpu+host"] = meas["gpu"]
        fastest = min(meas, key=meas.get)
        # online migration (Alg. 2): this buffer from the GPU placement to
        # GPU + host (half of it in HBM), one edp_migrate call, against the
        # makespan of its transfers run side by side (Appendix D, with the
        # flows fixed by the layout: the newer half HBM -> HBM, the older
        # half HBM -> page-locked memory)
        cfg2 = edp.make_config(self.cap, (self.C, self.H, self.W),
                               edp.EDP_XFORM_CHW_NORM_BF16, hbm_capacity=self.cap // 2,
                               tokens=self.L, norm_mean=MEAN3, norm_std=STD3,
                               device=device.index or 0)
        r2 = edp.Ring(cfg2, action=False, done=False)
        torch.cuda.synchronize()
        e0, e1 = mk(), mk()
        e0.record(stream)
        edp.edp_migrate(self.ring.ctx, r2.ctx)
        e1.record(stream)
        torch.cuda.synchronize()
        edp.edp_sync(r2.ctx)
        mig_s = e0.elapsed_time(e1) / 1e3
        n_h = self.cap // 2
        f_hbm, f_host = n_h * x, (self.cap - n_h) * x
        pred_s = max(f_hbm / bw["hbm_copy"], f_host / bw["d2h_pinned"])
        r2.close()
        del r2
        migration = {"from": "gpu", "to": "gpu+host (half in HBM)",
                     "bytes_to_hbm": f_hbm, "bytes_to_host": f_host,
                     "measured_ms": mig_s * 1e3, "predicted_makespan_ms": pred_s * 1e3}
        return {"migration": migration,
                "bandwidth_GBs": dict({k: v / 1e9 for k, v in bw.items() if k != "hbm_free"},
                                      host_gather_copy=bw_gather_copy / 1e9),
                "mem_GB": {"gpu": mem_gpu / 1e9, "host": mem_host / 1e9},
                "map_c_buf_1e6": [{"x_bytes": xx, "placement": names[c] if c < 4 else None}
                                  for xx, c in zip(xs, pmap)],
                "at_this_sample": {
                    "x_bytes": x, "c_buf": self.cap,
                    "predicted_us_per_sample": {n: t * 1e6 for n, t in zip(names, t_pred)},
                    "measured_us_per_sample": {n: t * 1e6 for n, t in meas.items()},
                    "chosen": names[best], "fastest_measured": fastest,
                    "measured_ranking": sorted(meas, key=meas.get),
                    "predicted_ranking": [names[i] for i in sorted(range(4),
                                                                   key=lambda i: (t_pred[i], i))]}}

    def cpu_setup(self, host_rows=None):
        """The oracle's host ring: by default at least 16 GB of images
        (110,000 rows, 16.6 GB), so its gathers miss the host caches as the
        GPU's miss L2; filled from one 256 MB random block (the timing does
        not depend on the byte values).  Capped at the capacity and at a
        quarter of the host's available memory."""
        import numpy as np
        import oracle as orc
        from paper_2609_24456_gb300 import fixtures as fx
        self.orc = orc
        if host_rows is None:
            host_rows = 110_000
            avail = _mem_available()
            if avail:
                host_rows = min(host_rows, int(avail // 4 // self.F))
        self.hrows = max(1, min(host_rows, self.cap))
        rng = np.random.default_rng(self.seed)
        block = rng.integers(0, 256, size=(min(self.hrows, max(1, (256 << 20) // self.F)),
                                           self.F), dtype=np.uint8)
        self.h_obs = np.empty((self.hrows, self.F), dtype=np.uint8)
        for lo in range(0, self.hrows, len(block)):
            n = min(len(block), self.hrows - lo)
            self.h_obs[lo:lo + n] = block[:n]
        self.h_tok, self.h_rew = fx.mm_metadata(self.seed, self.hrows, tokens=self.L)
        if self.ingest:
            self.h_stage = rng.integers(0, 256, size=(self.ingest, self.F), dtype=np.uint8)
            self.h_demoted = np.empty_like(self.h_stage)
        self.cpu_sample = ("per-step work of this workload (uniform B=%d, normalised bf16 "
                           "images, tokens, rewards%s) reading a %d-transition host ring "
                           "(%.1f GB)" % (self.B, ", ingest + demotion of %d" % self.ingest
                                          if self.ingest else "", self.hrows,
                                          self.hrows * self.F / 1e9))

    def cpu_round(self, r):
        orc = self.orc
        if self.ingest:  # demote the oldest rows, then write the new ones
            rows = (r * self.ingest + np.arange(self.ingest)) % self.hrows
            self.h_demoted[:] = self.h_obs[rows]
            self.h_obs[rows] = self.h_stage
        idx = orc.sample_uniform(self.cap, self.cap, self.cap, self.B, self.seed, r)
        orc.deliver_mm(self.h_obs, self.h_tok, self.h_rew, self.C, self.H * self.W,
                       idx % self.hrows, MEAN3, STD3)


class LlmBatch(Workload):
    """GRPO post-training batch (synthetic stand-in for a DAPO-Math-style
    rollout): 512 prompts x 16 responses of U[128, 4,096] tokens (~17.3 M
    int32 tokens), rewards 0/1 for half the groups and N(0, 1) for the rest.
    Step = group-relative advantages (ingestion) + the whole batch delivered
    in a shuffled order as packed tokens with output offsets and every token
    carrying its response's advantage (delivery)."""
    name = "grpo-batch-512x16-128..4096tok"
    kernel = "k_pack_gather"
    dtype = "i32,f32 (f64 group sums)"
    P, G = 512, 16

    def __init__(self, seed=1238, perms=8):
        import numpy as np
        self.seed, self.n_perm = seed, perms
        from paper_2609_24456_gb300 import fixtures as fx
        self.h_tok, self.h_off, self.h_r, self.h_goff = fx.llm_rollout(seed, self.P, self.G)
        self.n = len(self.h_r)
        # the delivery orders, on the host (the CPU legs use them too)
        rng = np.random.default_rng(self.seed)
        self.h_perms = [rng.permutation(self.n).astype(np.int64) for _ in range(self.n_perm)]
        self.T = int(self.h_off[-1])
        n, T = self.n, self.T
        grpo = 4 * n + 8 * (self.P + 1) + 4 * n
        # per sequence: idx 8, offsets 16, out offset 8, value 4; per token:
        # read 4, write 4 + 4
        self.deliver_bytes = n * (8 + 16 + 8 + 4) + 12 * T
        self.round_bytes = grpo + self.deliver_bytes
        self.launches_per_round = 2  # advantages + length pass, then the gather

    def config(self):
        return {"workload": self.name, "prompts": self.P, "responses_per_prompt": self.G,
                "tokens": self.T, "lengths": "U[128, 4096]",
                "l2": "token array 69 MB in, 138 MB out per step, rotating over 2 output sets"}

    def setup(self, device):
        import numpy as np
        import torch
        from paper_2609_24456_gb300 import edp
        self.edp = edp
        cfg = edp.make_config(64, (1, 16, 16), edp.EDP_XFORM_CHW_NORM_BF16,
                              device=device.index or 0)
        self.ring = edp.Ring(cfg, action=False, reward=False, done=False)
        self.tok = dev(self.h_tok, device)
        self.off = dev(self.h_off.view(np.int64), device)
        self.r = dev(self.h_r, device)
        self.goff = dev(self.h_goff.view(np.int64), device)
        self.adv = torch.empty(self.n, device=device)
        self.perms = [dev(p, device) for p in self.h_perms]
        self.outs = [(torch.empty(self.T, dtype=torch.int32, device=device),
                      torch.empty(self.T, device=device),
                      torch.empty(self.n + 1, dtype=torch.int64, device=device),
                      torch.empty(8 * (self.n // 8 + 1), dtype=torch.int64, device=device))
                     for _ in range(2)]
        # tokens of each eighth of each permutation (mini-batch deliveries)
        lens = np.diff(self.h_off.astype(np.int64))
        self.part_tokens = [lens[p].reshape(8, -1).sum(axis=1) for p in self.h_perms]

    def _grpo(self):
        self.edp.edp_grpo_advantage(self.ring.ctx, self.r, self.goff, self.P, 1e-6, self.adv)

    def _pack(self, r, parts=1):
        """One packed delivery of the permuted batch, or `parts` (8) of its
        mini-batches, each with its own offsets, one after the other in the
        output."""
        ot, ov, oo, oparts = self.outs[r % 2]
        k = r % self.n_perm
        if parts == 1:
            self.edp.edp_pack_deliver(self.ring.ctx, self.tok, self.off, self.n,
                                      self.perms[k], self.n, ot, oo, self.T,
                                      seq_value=self.adv, out_value=ov)
            return
        m, done = self.n // parts, 0
        for p in range(parts):
            nt = int(self.part_tokens[k][p])
            self.edp.edp_pack_deliver(self.ring.ctx, self.tok, self.off, self.n,
                                      self.perms[k][p * m:(p + 1) * m], m,
                                      ot[done:done + nt], oparts[p * (m + 1):(p + 1) * (m + 1)],
                                      nt, seq_value=self.adv, out_value=ov[done:done + nt])
            done += nt

    def round(self, r):
        self._grpo()
        self._pack(r)

    def round_fused(self, r):
        ot, ov, oo, _ = self.outs[r % 2]
        self.edp.edp_grpo_pack_deliver(self.ring.ctx, self.r, self.goff, self.P, 1e-6,
                                       self.adv, self.tok, self.off, self.n,
                                       self.perms[r % self.n_perm], self.n, ot, oo, self.T,
                                       out_value=ov)

    def round_parts(self, r):
        self._grpo()
        self._pack(r, 8)

    def schedules(self):
        return [("fused", self.round_fused, "edp_grpo_pack_deliver: advantages beside the "
                 "batch's length pass, then one packed delivery of all 8,192 responses"),
                ("batched", self.round, "advantages, then one packed delivery of all "
                 "8,192 responses (g_del = 1)"),
                ("per-minibatch", self.round_parts, "advantages, then 8 packed deliveries "
                 "of 1,024 responses (g_del = 1/8)")]

    def deliver_once(self, r):
        self._pack(r)

    def latency_step(self, r, ev_end):
        self.round_fused(r)
        ev_end.record()

    def e2e_setup(self, device):
        import torch
        self.h_in = torch.from_numpy(self.h_r.copy()).pin_memory()
        self.h_idx = [torch.from_numpy(p).pin_memory() for p in self.h_perms]
        self.h_tok_out = torch.empty(self.T, dtype=torch.int32, pin_memory=True)
        self.h_v_out = torch.empty(self.T, dtype=torch.float32, pin_memory=True)
        self.h_o_out = torch.empty(self.n + 1, dtype=torch.int64, pin_memory=True)
        self.h2d = 4 * self.n + 8 * self.n
        self.d2h = 8 * self.T + 8 * (self.n + 1)

    def e2e_round(self, r):
        """Rewards and the batch order in, the packed batch copied out (the
        packed delivery can write into page-locked host memory directly, but
        its 4-byte stores cross the host link slower than a copy: 176 vs
        267 GB/s end to end)."""
        self.r.copy_(self.h_in, non_blocking=True)
        self.perms[r % self.n_perm].copy_(self.h_idx[r % self.n_perm], non_blocking=True)
        self.round_fused(r)
        ot, ov, oo, _ = self.outs[r % 2]
        self.h_tok_out.copy_(ot, non_blocking=True)
        self.h_v_out.copy_(ov, non_blocking=True)
        self.h_o_out.copy_(oo, non_blocking=True)

    def cpu_setup(self):
        from oracle import llm
        self.llm = llm
        self.cpu_sample = "whole steps of this workload (GRPO advantages of 8,192 rewards, " \
                          "packing of ~17.3 M tokens)"

    def cpu_round(self, r):
        adv = self.llm.grpo_advantage(self.h_r, self.h_goff, 1e-6)
        self.llm.pack(self.h_tok, self.h_off, self.h_perms[r % self.n_perm], adv)


class ShardedPerReplay(PerReplay):
    """The prioritized replay sharded over the ranks (N > 1, Sec. 5.1's
    shared-GPU placement): every rank holds a 1,000,000-frame shard (its own
    content) and a learner that receives 512 samples of each global batch of
    512 N, drawn from the distribution over all shards' leaves.  Step = one
    sharded round (paper_2609_24456_gb300.shard.ShardedPer): shard totals
    all-gathered, targets routed to their owners, the owners' descents and
    deliveries, rows back to the learners, importance weights against the
    global minimum, TD-error updates back to the owners.  Rounds run eagerly:
    each waits on the host for its routing counts, which size the
    all-to-alls."""

    # total, routing, descent, delivery, batch minimum, weights, update
    launches_per_round = 7

    def __init__(self, rank=0, **kw):
        super().__init__(**kw)
        self.sample_seed = self.seed
        self.seed = self.seed + 7919 * rank  # this shard's content and TD errors

    def setup(self, device):
        from paper_2609_24456_gb300.shard import ShardComm, ShardedPer
        super().setup(device)
        self.sp = ShardedPer(self.ring, ShardComm(), self.B, beta=BETA, alpha=ALPHA, eps=EPS)

    def config(self):
        c = super().config()
        c.update(workload=self.name + "-sharded", batch_per_rank=self.B,
                 exchange="all-gather of shard totals, all-to-all of counts, targets, "
                          "rows and TD errors, min-reduce of the batch minimum")
        return c

    def round(self, r):
        self.sp.sample_deliver(self.sample_seed, r)
        self.sp.update(td=self.td[r % self.td_rounds])

    def schedules(self):
        return [("sharded", self.round, "sharded round, eager (host-sized exchanges)")]

    def time_latency(self, n, mk, stream):
        import torch
        out = []
        for r in range(n):
            e0, e1 = mk(), mk()
            e0.record(stream)
            self.sp.sample_deliver(self.sample_seed, 100000 + r)
            e1.record(stream)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) * 1e3)
        return out

    def e2e_setup(self, device):
        import torch
        lo = self.sp.out
        self.h_out = {k: torch.empty(lo[k].shape, dtype=lo[k].dtype, pin_memory=True)
                      for k in ("obs", "nxt", "isw", "idx")}
        self.h2d = 0
        self.d2h = sum(t.numel() * t.element_size() for t in self.h_out.values())

    def e2e_round(self, r):
        self.sp.sample_deliver(self.sample_seed, r)
        for k, t in self.h_out.items():
            t.copy_(self.sp.out[k], non_blocking=True)
        self.sp.update(td=self.td[r % self.td_rounds])


class ShardedPpoIteration(PpoIteration):
    """The on-policy iteration with environments sharded over the ranks
    (N > 1): every rank holds 256 environments x 128 steps; GAE per rank,
    the advantage normalisation over every rank's values (one fp64
    all-reduce of (n, sum A, sum A^2)), then the rank's shuffle and its 8
    mini-batches delivered in one call.  Eager."""

    def __init__(self, rank=0, **kw):
        super().__init__(**kw)
        self.seed = self.seed + 7919 * rank
        # scan, statistics, normalisation, shuffle (3), delivery
        self.launches_per_round = 7

    def setup(self, device):
        import torch
        from paper_2609_24456_gb300.shard import ShardComm
        self.comm = ShardComm()
        self.stats = torch.zeros(3, dtype=torch.float64, device=device)
        super().setup(device)

    def config(self):
        c = super().config()
        c.update(workload=self.name + "-sharded",
                 exchange="all-reduce of (n, sum A, sum A^2) in fp64")
        return c

    def _gae(self):
        from paper_2609_24456_gb300.shard import sharded_gae
        sharded_gae(self.ring.ctx, self.comm, self.r, self.v, self.d, self.T, self.E,
                    0.99, 0.95, self.adv, self.ret, self.nrm, self.stats)

    def round(self, r):
        self._gae()
        self.edp.edp_sample(self.ring.ctx, self.edp.EDP_SAMPLE_PERMUTE, self.n,
                            self.seed, r, self.idx)
        self._deliver_all(1)

    def schedules(self):
        return [("sharded", self.round, "sharded GAE normalisation, shuffle, one delivery "
                                        "call, eager")]

    def time_latency(self, n, mk, stream):
        import torch
        out = []
        for r in range(n):
            e0, e1 = mk(), mk()
            e0.record(stream)
            self.latency_step(100000 + r, e1)
            torch.cuda.synchronize()
            out.append(e0.elapsed_time(e1) * 1e3)
        return out

    def extra(self, device, mk, stream, deliver_us):
        return {}


# with N > 1 ranks these workloads run sharded (one exchange per step);
# the others run N independent replicas
SHARDED = {"per1m": ShardedPerReplay, "ppo": ShardedPpoIteration}

WORKLOADS = {
    "per1m": PerReplay,
    "dqn10k": DqnTiny,
    "ppo": PpoIteration,
    "mm200k": MmReplay,
    "grpo": LlmBatch,
    # two-tier: 1,600,000 transitions (~244 GB), newest half in HBM (122 GB),
    # oldest half in page-locked host memory (122 GB), 4,096 ingested per step
    "tiered": lambda **kw: MmReplay(capacity=kw.get("capacity") or 1_600_000,
                                    hbm_frac=0.5, ingest=4096),
}


# ----------------------------------------------------------------------------
def _mem_available():
    """MemAvailable of this host in bytes (0 if unknown)."""
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    return float(line.split()[1]) * 1024
    except OSError:
        pass
    return 0.0


def time_cpu(wl, budget_s, min_rounds=3):
    wl.cpu_round(0)
    n, t0 = 0, time.perf_counter()
    while n < min_rounds or time.perf_counter() - t0 < budget_s:
        wl.cpu_round(n + 1)
        n += 1
    dt = time.perf_counter() - t0
    return n, dt


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    wl = WORKLOADS[args.workload]()
    wl.cpu_setup()
    for r in range(args.warmup):
        wl.cpu_round(r)
    t0 = time.perf_counter()
    for r in range(args.steps):
        wl.cpu_round(args.warmup + r)
    dt = time.perf_counter() - t0
    gbs = wl.round_bytes * args.steps / dt / 1e9
    cores = oracle_threads()
    line = {"metric": "experience-delivery GB/s", "value": gbs, "unit": "GB/s",
            "impl": "reference", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": dt * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": wl.dtype, "data": "synthetic",
            "config": dict(wl.config(), parallelism="replicas%d" % int(
                os.environ.get("WORLD_SIZE", "1"))),
            "cpu_baseline": {"value": gbs, "unit": "GB/s", "cores": cores,
                             "kind": "oracle", "sample": wl.cpu_sample},
            "e2e": {"value": gbs, "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def job_ms(ms, dist, device):
    """Job time of a timed region: the maximum over ranks (every rank's
    replica must finish), or the local time with one rank."""
    if dist is None:
        return ms
    import torch
    on = device if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([ms], dtype=torch.float64, device=on)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_gbs(bytes_per_step, steps, world, ms):
    """Whole-job throughput: every rank processed `steps` units of
    `bytes_per_step` (weak scaling: fixed work per rank) in `ms`."""
    return bytes_per_step * steps * world / (ms / 1e3) / 1e9


def run_edp(args):
    import torch
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group(args.dist_backend)
    # one rank per GPU; with fewer GPUs than ranks (gloo, host-staged
    # exchanges) ranks share them
    local = local % max(1, torch.cuda.device_count())
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    from paper_2609_24456_gb300 import build
    # one rank per node compiles (if anything is stale); the others wait
    if local == 0:
        build.build()
    if dist:
        dist.barrier()
    build.build()  # up to date by now: only checks

    if args.workload == "ppo" and args.capacity:
        raise SystemExit("--capacity does not apply to the ppo workload")
    kw = {"capacity": args.capacity} if args.capacity else {}
    sharded = world > 1 and args.workload in SHARDED
    if sharded:
        wl = SHARDED[args.workload](rank=rank, **kw)
        args.no_graph = True  # every round sizes its exchanges on the host
    else:
        wl = WORKLOADS[args.workload](**kw)
    wl.setup(device)
    K, W = args.steps, args.warmup
    mk = lambda: torch.cuda.Event(enable_timing=True, external=True)
    stream = torch.cuda.current_stream()

    # warm-up rounds (eager), then capture the timed rounds in one graph;
    # no events inside it (event nodes split the graph and cost several us)
    scheds = wl.schedules()
    if args.schedule:
        names = [n for n, _, _ in scheds]
        if args.schedule not in names:
            raise SystemExit("--schedule: one of %s" % names)
        scheds.sort(key=lambda x: x[0] != args.schedule)

    def rounds(first, n, fn):
        for r in range(first, first + n):
            fn(r)
        wl.join()

    def timed(fn):
        rounds(K, W, fn)
        torch.cuda.synchronize()
        g = None
        if not args.no_graph:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, capture_error_mode="thread_local"):
                rounds(0, K, fn)
            g.replay()  # upload + warm the graph (rounds are re-timed below)
            torch.cuda.synchronize()
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        clocks = Clocks(local)
        clocks.start()
        time.sleep(0.02)
        t_start, t_end = mk(), mk()
        t_start.record(stream)
        g.replay() if g is not None else rounds(0, K, fn)
        t_end.record(stream)
        torch.cuda.synchronize()
        clk = clocks.stop()
        return job_ms(t_start.elapsed_time(t_end), dist, device), clk

    use_graph = not args.no_graph
    others = []
    for name, fn, desc in ([] if args.no_other_schedules else scheds[1:]):
        ms_o, _ = timed(fn)
        others.append({"schedule": name, "value": job_gbs(wl.round_bytes, K, world, ms_o),
                       "ms_per_step": ms_o / K, "description": desc})
    ms, clk = timed(scheds[0][1])
    ms_step = ms / K
    value = job_gbs(wl.round_bytes, K, world, ms)
    peak, peak_kind = peaks()

    # dominant kernel: the fused delivery, timed back to back on the same
    # stream (events bracket the launches; the batches are real samples)
    Kd = min(K, args.kernel_steps)
    deliver_us = wl.time_deliver(Kd, mk, stream, graph=use_graph)
    # p50 sample -> batch latency: events before sampling and after delivery
    Kl = min(K, args.latency_steps)
    lat_us = sorted(wl.time_latency(Kl, mk, stream))
    p50 = lat_us[len(lat_us) // 2]

    # end-to-end through the C ABI with host buffers (eager calls)
    e2e = None
    if not args.no_e2e:
        wl.e2e_setup(device)
        Ke = min(K, args.e2e_steps)
        for r in range(3):
            wl.e2e_round(r)
        wl.join()
        torch.cuda.synchronize()
        if dist:
            dist.barrier()
        e0, e1 = mk(), mk()
        e0.record(stream)
        for r in range(Ke):
            wl.e2e_round(r)
        wl.join()  # side streams a schedule used
        e1.record(stream)
        torch.cuda.synchronize()
        ems = job_ms(e0.elapsed_time(e1), dist, device)
        e2e = {"value": job_gbs(wl.round_bytes, Ke, world, ems),
               "unit": "GB/s", "h2d_bytes_per_step": wl.h2d,
               "d2h_bytes_per_step": wl.d2h, "steps": Ke,
               "ms_per_step": ems / Ke}

    avg_deliver_s = deliver_us / 1e6
    achieved = wl.deliver_bytes / avg_deliver_s / 1e9
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak,
                "unit": "GB/s", "frac": achieved / peak, "peak_kind": peak_kind,
                "kernel": wl.kernel,
                "traffic": kernel_traffic(wl.kernel, wl.name),
                "algorithmic_bytes_per_launch": wl.deliver_bytes,
                "avg_launch_us": avg_deliver_s * 1e6, "launches_timed": Kd}
    if getattr(wl, "tiered", False):
        # the HBM fraction understates this launch: its host-tier share is
        # read over the host link, whose fraction host_link reports
        roofline["note"] = ("two-tier: %.0f%% of the samples are read over the host link; "
                            "see host_link.frac_of_link" % (100.0 * (wl.cap - wl.cap_h) / wl.cap))

    extra = {}
    if hasattr(wl, "extra") and not args.no_extra:
        extra = wl.extra(device, mk, stream, deliver_us)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        wl.cpu_setup()
        n, dt = time_cpu(wl, args.cpu_seconds)
        cores = oracle_threads()
        cpu = {"value": wl.round_bytes * n / dt / 1e9, "unit": "GB/s",
               "cores": cores, "kind": "oracle",
               "sample": "%d rounds: %s" % (n, wl.cpu_sample)}
        # the same oracle on one core (a shorter sample)
        oracle_set_threads(1)
        n1, dt1 = time_cpu(wl, max(1.0, args.cpu_seconds / 3))
        oracle_set_threads(cores)
        cpu["single_thread"] = {"value": wl.round_bytes * n1 / dt1 / 1e9, "unit": "GB/s",
                                "cores": 1, "sample": "%d rounds" % n1}

    if rank == 0:
        line = {"metric": "experience-delivery GB/s", "value": value,
                "unit": "GB/s", "n_gpus": world, "steps": K, "warmup": W,
                "ms_per_step": ms_step, "higher_is_better": True,
                "scaling": "weak", "vs_baseline": None, "dtype": wl.dtype,
                "data": "synthetic",
                # the workload alone, as the reference arm prints it; how it
                # ran goes beside it
                "config": dict(wl.config(), parallelism=("sharded%d" if sharded
                                                         else "replicas%d") % world),
                "schedule": "%s: %s" % scheds[0][::2], "graph": use_graph,
                "pct_hbm_peak": 100.0 * value / peak,
                "batches_per_s": K * world / (ms / 1e3),
                "p50_sample_to_batch_us": p50,
                "roofline": roofline, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": wl.launches_by_schedule.get(scheds[0][0],
                                                            wl.launches_per_round) * K,
                "clocks": clk}
        if others:
            line["other_schedules"] = others
        split = wl.split_bytes() if hasattr(wl, "split_bytes") else None
        if split:  # HBM and host-link throughput of the step, separately
            line["split_GBs"] = {k: v * K * world / (ms / 1e3) / 1e9 for k, v in split.items()}
        line.update(extra)
        print(json.dumps(line))
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="edp", choices=["edp", "reference"])
    ap.add_argument("--dist-backend", default="nccl", choices=["nccl", "gloo"],
                    help="process-group backend for N > 1 (gloo stages the sharded "
                         "exchanges through host memory, so several ranks may share a GPU)")
    # default: the largest HBM-resident configuration (200,000 multimodal
    # transitions, ~30 GB), whose metric is the fraction of HBM bandwidth
    ap.add_argument("--workload", default="mm200k", choices=sorted(WORKLOADS))
    ap.add_argument("--capacity", type=int, default=0,
                    help="override the ring capacity (profiling small cases)")
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-other-schedules", action="store_true",
                    help="time only the main schedule")
    ap.add_argument("--schedule", default="",
                    help="the workload's schedule timed as the main number "
                         "(default: its first); the others are reported too")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the workload's side measurements (ingest timing, "
                         "scheduling and placement experiments)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--e2e-steps", type=int, default=200)
    ap.add_argument("--kernel-steps", type=int, default=500)
    ap.add_argument("--latency-steps", type=int, default=200)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        return run_reference(args)
    return run_edp(args)


if __name__ == "__main__":
    sys.exit(main())
