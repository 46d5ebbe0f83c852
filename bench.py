"""Benchmark of the frontier-accounting hot path on GB300.

One step = one pass of the whole path over one batch of synthetic telemetry:
per-rank window medians, then one evidence pass that computes the frontier
(Sec. 3 Eq. 1), the window aggregates with lead-rank credit (Eq. 2) and the
clipped-gain numerators (Sec. 4 Eq. 4), then top-k suspects and the App. C
gates.  The standalone frontier/aggregation pass (sf_window_aggregate) is timed
beside the step as `frontier_pass`.  The default workload is the largest
frontier-accounting configuration: 8192 ranks x 8 stages x 20000 steps of
int64 ns (10.49 GB), 1000-step windows, top-5, labels.

Prints ONE JSON line (rank 0).  `value` is rank.step.stage records per
second with the input resident in HBM (CUDA events on the launching stream,
max over ranks); `e2e` is the same metric through the library's public API
with the input in pinned host memory and its host->device copy (plus the
device->host read of the results) inside the timed region.  `roofline` is
the dominant kernel's algorithmic HBM bytes over its event-timed duration
against the measured copy bandwidth.  `cpu_baseline` times the CPU oracle on
a bounded sample of the same workload.

Multi-GPU (torchrun): one independent replica per GPU (the path has no
exchange step), weak scaling, barrier + max-over-ranks timing.
`--impl reference` times the CPU oracle itself as the reference arm.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from synth import workloads as wl  # noqa: E402

METRIC = "rank·step·stage records/sec and achieved HBM GB/s (% of GB300 peak)"
UNIT = "records/s"
# the sources each roofline kernel is compiled from: a recorded DRAM traffic
# figure is valid only while their hash is the one it was captured with
KERNEL_SOURCES = {"window_median": ("sf_select.cu", "sf_device.cuh"),
                  "direct_gain": ("sf_stream.cu", "sf_device.cuh")}


# --------------------------------------------------------------------------- distributed harness

def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def init_dist(backend: str):
    ws, rank, _ = dist_env()
    if ws > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group(backend=backend)
    return ws, rank


def barrier(ws: int):
    if ws > 1:
        torch.distributed.barrier()


def max_over_ranks(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


# Device-side delay queued before the first timed event when `ahead` is set:
# about 10 ms at the GB300's 2 GHz SM clock, longer than the host needs to
# enqueue 20 steps of a few launches each.
AHEAD_CYCLES = 20_000_000
L2_FLUSH_BYTES = 256 << 20  # a read of twice the 129 MB L2 evicts every input line


NOMINAL_HBM_GBS = 8000.0  # GB300 HBM3e, nominal


def add_nominal(rec, peak: float, peak_kind: str):
    """Beside every `frac` (achieved GB/s over the measured copy bandwidth,
    which counts read and write bytes, so read-mostly passes can exceed 1),
    add `frac_nominal`: the same GB/s over the nominal HBM3e rate."""
    if isinstance(rec, dict):
        gbs = rec.get("gbs", rec.get("achieved"))
        if "frac" in rec and isinstance(gbs, (int, float)):
            rec["frac_nominal"] = round(gbs / NOMINAL_HBM_GBS, 4)
        for v in rec.values():
            add_nominal(v, peak, peak_kind)
    elif isinstance(rec, list):
        for v in rec:
            add_nominal(v, peak, peak_kind)
    return rec


def peaks_record(peak: float, peak_kind: str) -> dict:
    return {"frac": f"of the {peak_kind} copy bandwidth {peak} GB/s (read + write bytes of a device copy)",
            "frac_nominal": f"of the nominal HBM3e rate {NOMINAL_HBM_GBS:.0f} GB/s"}


def timed_loop(step, K: int, W: int, ws: int, device, use_cuda: bool, ahead: bool = False) -> float:
    """Run W untimed then K timed steps; returns the max-over-ranks seconds.

    ahead: queue the K steps behind a device-side delay, so that the events
    bracket back-to-back device execution even when one step's kernels take
    less time than the host needs to launch them (launches of ~10-30 us on
    inputs of a few MB); the delay itself lies before the first event."""
    for _ in range(W):
        step()
    if use_cuda:
        torch.cuda.synchronize()
    barrier(ws)
    if use_cuda:
        stream = torch.cuda.current_stream()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        if ahead:
            torch.cuda._sleep(AHEAD_CYCLES)
        e0.record(stream)
        for _ in range(K):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
        secs = e0.elapsed_time(e1) / 1e3
    else:
        t0 = time.perf_counter()
        for _ in range(K):
            step()
        secs = time.perf_counter() - t0
    barrier(ws)
    return max_over_ranks(secs, ws, device)


def timed_loop_flushed(step, K: int, W: int, device) -> float:
    """K steps on an input smaller than L2, each preceded by a read of
    L2_FLUSH_BYTES so that it reads its input from HBM (a read, not a write:
    the evicting lines are clean, so no write-back of the flush runs under
    the timed step); a pair of events brackets each step alone, and
    everything is queued behind a device-side delay so that no host gap
    falls inside a pair.  Returns the summed seconds of the K steps (one GPU)."""
    scratch = torch.ones(L2_FLUSH_BYTES // 4, dtype=torch.int32, device=device)
    for _ in range(W):
        scratch.sum()
        step()
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    torch.cuda._sleep(AHEAD_CYCLES)
    for i in range(K):
        scratch.sum()
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    secs = sum(a.elapsed_time(b) for a, b in ev) / 1e3
    del scratch
    return secs


# --------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu = gpu_id
        self.proc = None
        # raw samples go to SF_CLOCKS_DIR (default: the system temp directory)
        self.path = os.path.join(os.environ.get("SF_CLOCKS_DIR", tempfile.gettempdir()), f"clocks_gpu{os.getpid()}.csv")

    def __enter__(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except OSError:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                smax = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------- helpers

def smi_gpu_id(local: int) -> str:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [v.strip() for v in vis.split(",") if v.strip()]
        if local < len(ids):
            return ids[local]
    return str(local)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def kernel_source_sha(kernel: str) -> str:
    h = hashlib.sha256()
    for f in KERNEL_SOURCES.get(kernel, ("sf_stream.cu", "sf_select.cu", "sf_device.cuh")):
        with open(os.path.join(ROOT, "paper_2606_06751_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch recorded from an ncu capture in profiles/, valid
    only while the kernel sources are unchanged (matching source sha)."""
    sha = kernel_source_sha(kernel)
    pdir = os.path.join(ROOT, "profiles")
    if not os.path.isdir(pdir):
        return None
    for fn in sorted(os.listdir(pdir)):
        if not fn.endswith(".md"):
            continue
        txt = open(os.path.join(pdir, fn)).read()
        for m in re.finditer(r"traffic_per_launch\s+kernel=(\S+)\s+workload=(\S+)\s+bytes=(\d+)\s+"
                             r"source_sha=(\S+)", txt):
            if m.group(1) == kernel and m.group(2) == workload and m.group(4) == sha:
                return int(m.group(3))
    return None


# --------------------------------------------------------------------------- our arm

class Pipeline:
    """Device buffers and the per-step sequence of library calls."""

    def __init__(self, sf, w: wl.Workload, d: torch.Tensor):
        self.sf, self.w, self.d = sf, w, d
        dev = d.device
        T, R, S, W, k = w.T, w.R, w.S, w.W, w.k
        self.nW = sf.num_windows(0, T, W)
        nW = self.nW
        e = lambda shape, dt: torch.empty(shape, dtype=dt, device=dev)  # noqa: E731
        self.top = sf.TopK(e((nW, k), torch.int32), e((nW, k), torch.int64), e((nW, k, 2), torch.int32),
                           e((nW, k), torch.int64))
        self.m = e((nW, R, S), torch.int64)
        self.ev = sf.Evidence(e((nW, S), torch.int64), e((nW, S), torch.int64), e((nW,), torch.int64),
                              e((T,), torch.uint8), None, e((nW, S, R), torch.int64), e((nW, S, R), torch.int32))
        self.lab = sf.Labels(e((nW,), torch.int32), e((nW,), torch.int32), e((nW,), torch.int32),
                             e((nW, S), torch.float64), e((nW, S), torch.float64), e((nW,), torch.int32),
                             e((nW,), torch.int32))
        self.win = sf.Windows(e((nW, S), torch.int64), e((nW,), torch.int64), e((nW, S, R), torch.int64),
                              e((nW, S, R), torch.int32), e((T,), torch.uint8))
        self.base = sf.Baselines(e((nW, S), torch.int64), e((nW, S, 2), torch.uint64), e((nW, S), torch.int64),
                                 e((nW, S), torch.int64))
        self.lag = sf.Lag(e((T, S), torch.int64), e((T, S), torch.int64), e((T, S), torch.int64))
        self.spread = e((nW, S), torch.int64)
        self.fr_a = e((T, S), torch.int64)    # frontier increments, input of the tie-set pass
        self.ties = e((T, S), torch.int32)
        self.rank_ws = sf.rank_workspace(T, R, S, dev)
        # role groups: nodes of 128 consecutive ranks (one group when R <= 128)
        self.n_groups = max(1, R // 128)
        self.node_group = (torch.arange(R, device=dev, dtype=torch.int32) * self.n_groups // R).to(torch.int32)
        self.grp = sf.GroupWindows(e((nW, self.n_groups, S), torch.int64), e((nW, self.n_groups), torch.int64))
        self.status = sf.new_status(dev)
        self.names = ["window_median", "direct_gain", "topk_suspects", "label_gates"]
        self.events = None

    def step(self, d=None, timing=False):
        sf, w = self.sf, self.w
        d = self.d if d is None else d
        ev = None
        if timing:
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(5)]
            ev[0].record()
        sf.sf_window_median(d, w.W, m=self.m, status=self.status)
        if timing:
            ev[1].record()
        sf.sf_direct_gain(d, w.W, self.m, out=self.ev, status=self.status)
        if timing:
            ev[2].record()
        sf.sf_topk_suspects(self.ev.X, self.ev.E, w.k, out=self.top)
        if timing:
            ev[3].record()
        sf.sf_label_gates(w.T, w.R, w.S, w.W, self.ev, out=self.lab)
        if timing:
            ev[4].record()
            self.events.append(ev)

    def aggregate(self):
        """The standalone frontier pass with window aggregation (sf_window_aggregate)."""
        self.sf.sf_window_aggregate(self.d, self.w.W, X=self.win.X, D=self.win.D, E=self.win.E, C=self.win.C,
                                    step_lead=self.win.step_lead, status=self.status)

    def baselines(self):
        """The routing-baseline pass (sf_window_baselines)."""
        self.sf.sf_window_baselines(self.d, self.w.W, out=self.base, status=self.status)

    def rank_lag(self):
        """The cross-rank lag / delta-lag / gap pass (sf_rank_lag)."""
        self.sf.sf_rank_lag(self.d, out=self.lag, workspace=self.rank_ws, status=self.status)

    def raw_spread(self):
        """The raw rank spread per window (sf_raw_spread)."""
        self.sf.sf_raw_spread(self.d, self.w.W, spread=self.spread, workspace=self.rank_ws, status=self.status)

    def frontier_ties(self):
        """Size of the lead rank's tie set per step and stage (sf_frontier_ties),
        on the increments of an earlier sf_frontier call."""
        self.sf.sf_frontier_ties(self.d, a=self.fr_a, ties=self.ties, status=self.status)

    def group_aggregate(self):
        """The frontier within node groups of 128 ranks (sf_group_aggregate)."""
        self.sf.sf_group_aggregate(self.d, self.node_group, self.n_groups, self.w.W, out=self.grp,
                                   status=self.status)

    def results(self):
        return [self.lab.labels, self.lab.route_mask, self.lab.amb_mask, self.lab.share, self.lab.gain,
                self.top.stage, self.top.pair, self.top.pair_value, self.ev.X, self.ev.D]

    def algorithmic_bytes(self):
        w, nW = self.w, self.nW
        din = w.T * w.R * w.S * 8
        return {
            "window_median": din + nW * w.R * w.S * 8,
            "direct_gain": din + nW * w.R * w.S * 8 + nW * w.S * (w.R * 12 + 16) + nW * 8 + w.T,
            "topk_suspects": nW * w.S * (w.R + 1) * 8 + nW * w.k * 24,
            "label_gates": nW * (2 * w.S + 1) * 8 + w.T + nW * (3 * 4 + 2 * w.S * 8),
            "window_aggregate": din + nW * w.S * (w.R * 12 + 8) + nW * 8 + w.T,
            "window_baselines": din + nW * w.S * 40 + w.T * w.S * 16,
            "rank_lag": din + 3 * w.T * w.S * 8,
            "raw_spread": din + nW * w.S * 8,
            "group_aggregate": din + w.R * 4 + nW * self.n_groups * (w.S + 1) * 8,
            "frontier_ties": din + w.T * w.S * (8 + 4),
        }


def run_ours(args):
    ws, rank, local = dist_env()
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    init_dist("nccl")
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_06751_gb300 import stagefrontier as sf

    w = wl.by_name(args.workload, seed=args.seed + rank, steps=args.steps_override)
    host = torch.empty((w.T, w.R, w.S), dtype=torch.int64, pin_memory=True)
    w.fill(host.numpy().reshape(-1), threads=max(1, (os.cpu_count() or 1) // ws))
    d = torch.empty_like(host, device=device)
    d.copy_(host)
    torch.cuda.synchronize()
    pipe = Pipeline(sf, w, d)
    records = w.records

    # device-resident timing, clocks sampled throughout
    pipe.events = []
    n0 = sf.launch_count()
    with ClockSampler(smi_gpu_id(local)) as clk:
        secs = timed_loop(lambda: pipe.step(timing=True), args.steps, args.warmup, ws, device, True)
    launches = sf.launch_count() - n0
    torch.cuda.synchronize()
    st = int(pipe.status.item())
    if st != 0:
        raise RuntimeError(f"device status {st} during the timed region")
    timed = pipe.events[args.warmup:]
    per_kernel = {n: [] for n in pipe.names}
    for ev in timed:
        for i, n in enumerate(pipe.names):
            per_kernel[n].append(ev[i].elapsed_time(ev[i + 1]) / 1e3)
    # median over the timed steps: robust to the first step, which follows a
    # synchronize and so also carries the host's enqueue latency
    avg = {n: statistics.median(v) for n, v in per_kernel.items()}
    algo = pipe.algorithmic_bytes()
    dominant = max(avg, key=avg.get)
    peak, peak_kind = peaks()
    achieved = algo[dominant] / avg[dominant] / 1e9
    value = records * ws * args.steps / secs

    # the standalone frontier/aggregation pass and the routing-baseline pass, each timed on its own
    agg_secs = timed_loop(pipe.aggregate, args.steps, args.warmup, ws, device, True) / args.steps
    base_secs = timed_loop(pipe.baselines, args.steps, args.warmup, ws, device, True) / args.steps
    lag_secs = timed_loop(pipe.rank_lag, args.steps, args.warmup, ws, device, True) / args.steps
    spread_secs = timed_loop(pipe.raw_spread, args.steps, args.warmup, ws, device, True) / args.steps
    group_secs = timed_loop(pipe.group_aggregate, args.steps, args.warmup, ws, device, True) / args.steps
    sf.sf_frontier(d, a=pipe.fr_a, status=pipe.status, outputs=("a",))
    ties_secs = timed_loop(pipe.frontier_ties, args.steps, args.warmup, ws, device, True) / args.steps

    # rank-major ingest: the same steps as the gather delivers them (one
    # [R][n][S] block per window), converted back into d in place of itself
    def fill_gathered(x, out):
        """out (flat) <- x [T][R][S] in the gather's layout, block by block."""
        nfull, tail = w.T // w.W, w.T % w.W
        n = nfull * w.W * w.R * w.S
        out[:n].view(nfull, w.R, w.W, w.S).copy_(x[:nfull * w.W].view(nfull, w.W, w.R, w.S).permute(0, 2, 1, 3))
        if tail:
            out[n:].view(w.R, tail, w.S).copy_(x[nfull * w.W:].permute(1, 0, 2))
        return out

    g_dev = fill_gathered(d, torch.empty(w.T * w.R * w.S, dtype=torch.int64, device=device))
    ingest_secs = timed_loop(lambda: sf.sf_gathered_to_steps(g_dev, w.T, w.R, w.S, w.W, dst=d), args.steps,
                             args.warmup, ws, device, True) / args.steps
    del g_dev

    # every other configuration (the three smaller workloads and the twelve
    # 1 GiB sweep shapes): frontier and aggregation passes and the whole step
    # on the GPU, the oracle on a bounded sample single-threaded and on all cores
    configs = None
    if ws == 1 and not args.no_configs:
        from oracle import oracle as O
        O.build_lib()
        configs = [measure_config(n, sf, device, peak, 5, 3, args.seed, oracle=O)
                   for n in CONFIG_NAMES + FEW_STEP_NAMES + GENERIC_NAMES if n != w.name]

    # end to end through the host-memory entry point: every step streams the
    # pinned host tensor to the GPU in 2000-step chunks (copies overlapping the
    # previous chunk's compute) and reads the per-window results back
    chunk = w.chunk_steps or w.T
    bufs = sf.StreamBuffers(w.T, w.R, w.S, w.W, w.k, chunk, device)
    copy_stream = torch.cuda.Stream(device)
    del d, pipe.d
    torch.cuda.empty_cache()
    outs = [bufs.out.labels, bufs.out.route_mask, bufs.out.amb_mask, bufs.out.share, bufs.out.gain,
            bufs.out.top_stage, bufs.out.top_pair, bufs.out.top_pair_value, bufs.out.X, bufs.out.D]
    host_outs = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs]
    d2h = sum(o.numel() * o.element_size() for o in outs)

    def e2e_step():
        sf.sf_stream_windows(host, w.W, w.k, chunk, bufs=bufs, status=pipe.status, copy_stream=copy_stream)
        for hb, o in zip(host_outs, outs):
            hb.copy_(o, non_blocking=True)

    # the host link's own rate for the same bytes: plain pinned copies of the
    # same chunks into one device buffer, timed before and after the e2e legs
    # (the link is shared with the machine's other tenants and drifts)
    link_buf = torch.empty((chunk, w.R, w.S), dtype=torch.int64, device=device)

    def link_pass():
        for c0 in range(0, w.T, chunk):
            n = min(chunk, w.T - c0)
            link_buf[:n].copy_(host[c0:c0 + n], non_blocking=True)

    link_steps = 5
    link_before = w.nbytes * ws * link_steps / timed_loop(link_pass, link_steps, 3, ws, device, True) / 1e9

    e2e_steps = max(20, args.steps)
    e2e_secs = timed_loop(e2e_step, e2e_steps, args.warmup, ws, device, True)
    e2e_value = records * ws * e2e_steps / e2e_secs

    # the same end to end over host telemetry in the gather's rank-major layout
    g_host = fill_gathered(host, torch.empty(w.T * w.R * w.S, dtype=torch.int64, pin_memory=True))
    gbufs = sf.StreamBuffers(w.T, w.R, w.S, w.W, w.k, chunk, device, gathered=True)

    def e2e_gathered_step():
        sf.sf_stream_gathered_windows(g_host, w.T, w.R, w.S, w.W, w.k, chunk, bufs=gbufs, status=pipe.status,
                                      copy_stream=copy_stream)
        for hb, o in zip(host_outs, [getattr(gbufs.out, n) for n in ("labels", "route_mask", "amb_mask", "share",
                                                                      "gain", "top_stage", "top_pair",
                                                                      "top_pair_value", "X", "D")]):
            hb.copy_(o, non_blocking=True)

    e2e_g_secs = timed_loop(e2e_gathered_step, e2e_steps, args.warmup, ws, device, True)
    link_after = w.nbytes * ws * link_steps / timed_loop(link_pass, link_steps, 3, ws, device, True) / 1e9
    link_gbs = (link_before + link_after) / 2
    # the gathered leg reads another pinned buffer, whose pages can sit
    # elsewhere in host memory: its own link rate, measured the same way
    g_flat = g_host.view(-1)
    link_flat = link_buf.view(-1)

    def link_pass_gathered():
        step_words = w.R * w.S
        for c0 in range(0, w.T, chunk):
            n = min(chunk, w.T - c0) * step_words
            link_flat[:n].copy_(g_flat[c0 * step_words:c0 * step_words + n], non_blocking=True)

    link_g_gbs = w.nbytes * ws * link_steps / timed_loop(link_pass_gathered, link_steps, 3, ws, device, True) / 1e9
    del gbufs, g_host, g_flat, link_flat, link_buf
    if int(pipe.status.item()) != 0:
        raise RuntimeError("device status set during the end-to-end loop")

    if rank != 0:
        return None
    kernels = {n: {"ms": round(avg[n] * 1e3, 4), "gbs": round(algo[n] / avg[n] / 1e9, 1),
                   "algorithmic_bytes": algo[n]} for n in pipe.names}
    agg_gbs = algo["window_aggregate"] / agg_secs / 1e9
    traffic = profiled_traffic(dominant, w.name)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
        "config": workload_config(w, args, ws),
        "step_gbs": sum(algo[n] for n in pipe.names) / (secs / args.steps) / 1e9,
        "roofline": {"kernel": dominant, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "traffic": traffic},
        "kernels": kernels,
        "frontier_pass": {"entry": "sf_window_aggregate", "ms": round(agg_secs * 1e3, 4),
                          "gbs": round(agg_gbs, 1), "frac": round(agg_gbs / peak, 4),
                          "records_per_s": records / agg_secs},
        "baselines_pass": {"entry": "sf_window_baselines", "ms": round(base_secs * 1e3, 4),
                           "gbs": round(algo["window_baselines"] / base_secs / 1e9, 1),
                           "frac": round(algo["window_baselines"] / base_secs / 1e9 / peak, 4)},
        "lag_pass": {"entry": "sf_rank_lag", "ms": round(lag_secs * 1e3, 4),
                     "gbs": round(algo["rank_lag"] / lag_secs / 1e9, 1),
                     "frac": round(algo["rank_lag"] / lag_secs / 1e9 / peak, 4)},
        "spread_pass": {"entry": "sf_raw_spread", "ms": round(spread_secs * 1e3, 4),
                        "gbs": round(algo["raw_spread"] / spread_secs / 1e9, 1),
                        "frac": round(algo["raw_spread"] / spread_secs / 1e9 / peak, 4)},
        "group_pass": {"entry": "sf_group_aggregate", "groups": pipe.n_groups, "ms": round(group_secs * 1e3, 4),
                       "gbs": round(algo["group_aggregate"] / group_secs / 1e9, 1),
                       "frac": round(algo["group_aggregate"] / group_secs / 1e9 / peak, 4)},
        "ties_pass": {"entry": "sf_frontier_ties", "ms": round(ties_secs * 1e3, 4),
                      "gbs": round(algo["frontier_ties"] / ties_secs / 1e9, 1),
                      "frac": round(algo["frontier_ties"] / ties_secs / 1e9 / peak, 4)},
        "ingest_pass": {"entry": "sf_gathered_to_steps", "ms": round(ingest_secs * 1e3, 4),
                        "gbs": round(2 * w.nbytes / ingest_secs / 1e9, 1),
                        "frac": round(2 * w.nbytes / ingest_secs / 1e9 / peak, 4)},
        "e2e_gathered": {"value": records * ws * e2e_steps / e2e_g_secs, "unit": UNIT,
                         "entry": "sf_stream_gathered_windows", "h2d_bytes_per_step": w.nbytes,
                         "steps": e2e_steps, "h2d_gbs": round(w.nbytes * ws * e2e_steps / e2e_g_secs / 1e9, 1),
                         "link_gbs": round(link_g_gbs, 1),
                         "frac_of_link": round(w.nbytes * ws * e2e_steps / e2e_g_secs / 1e9 / link_g_gbs, 3)},
        "gpu_launches": int(launches * args.steps // (args.steps + args.warmup)),
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": w.nbytes, "d2h_bytes_per_step": d2h,
                "entry": "sf_stream_windows", "chunk_steps": chunk, "steps": e2e_steps,
                "h2d_gbs": round(w.nbytes * ws * e2e_steps / e2e_secs / 1e9, 1),
                "link_gbs": round(link_gbs, 1), "link_gbs_before_after": [round(link_before, 1), round(link_after, 1)],
                "frac_of_link": round(w.nbytes * ws * e2e_steps / e2e_secs / 1e9 / link_gbs, 3)},
        "clocks": clk.summary(),
    }
    if configs is not None:
        line["configs"] = configs
    if ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_sample_windows)
    line["peaks"] = peaks_record(peak, peak_kind)
    return add_nominal(line, peak, peak_kind)


# --------------------------------------------------------------------------- oracle arm

def oracle_step(O, w: wl.Workload, d_np: np.ndarray):
    """The whole hot path on the CPU oracle, as it stands."""
    win = O.windows(d_np, w.W)
    O.topk(win.X, win.E, w.k)
    O.label_windows(d_np, w.W)


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo), for the report."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part")):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return "unknown"


def oracle_rate(O, w: wl.Workload, n: int, threads: int) -> dict:
    """The oracle on `threads` disjoint slices of n steps each (slice i: steps
    [i n, (i+1) n) of the workload, windows of min(W, n) steps), one host
    thread per slice (the C oracle releases the GIL).  Returns records/s over
    the wall time of all slices together."""
    from concurrent.futures import ThreadPoolExecutor
    n = max(1, min(n, w.T // threads))
    wn = min(w.W, n)
    slices = [w.generate(t0=i * n, nsteps=n) for i in range(threads)]
    sw = wl.Workload(**{**w.__dict__, "T": n, "W": wn})
    t0 = time.perf_counter()
    if threads == 1:
        oracle_step(O, sw, slices[0])
    else:
        with ThreadPoolExecutor(threads) as ex:
            list(ex.map(lambda x: oracle_step(O, sw, x), slices))
    secs = time.perf_counter() - t0
    rec = threads * n * w.R * w.S
    return {"value": rec / secs, "unit": UNIT, "cores": threads, "kind": "oracle", "secs": round(secs, 2),
            "sample": f"{threads} x {n} steps of {w.name} (windows of {wn}): {rec} records"}


def cpu_baseline(w: wl.Workload, n_windows: int):
    """The CPU oracle on the host's cores: single-threaded on the first
    n_windows windows, and on all cores over disjoint window ranges."""
    from oracle import oracle as O
    n = min(w.T, n_windows * w.W)
    one = oracle_rate(O, w, n, 1)
    cores = os.cpu_count() or 1
    per = max(w.W, (w.T // cores) // w.W * w.W)  # whole windows per thread, all of T at most
    threads = max(1, min(cores, w.T // per))
    allc = oracle_rate(O, w, per, threads)
    return {"value": one["value"], "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"first {n} steps ({n // w.W} windows) of {w.name}: {n * w.R * w.S} records, "
                      f"{one['secs']} s single-threaded C oracle (frontier/windows, top-k, medians, gains, gates)",
            "all_cores": {"value": allc["value"], "cores": allc["cores"], "sample": allc["sample"],
                          "secs": allc["secs"]},
            "host_cpus": cores, "cpu_model": cpu_model()}


def workload_config(w: wl.Workload, args, ws: int) -> dict:
    """The `config` object of the JSON line (the same for both arms)."""
    return {"workload": f"{w.name}: {w.R} ranks x {w.S} stages x {w.T} steps int64 ns "
                        f"({w.nbytes / 1e9:.2f} GB), windows of {w.W}, top-{w.k}, labels",
            "R": w.R, "S": w.S, "T": w.T, "W": w.W, "k": w.k, "seed": args.seed,
            "l2": f"input {w.nbytes / 1e9:.1f} GB > 129 MB L2 on every pass; no flush",
            "parallelism": "replicas" if ws > 1 else "single"}


def run_reference(args):
    """The CPU oracle as the reference arm: each step runs the whole hot path
    (frontier and windows, top-k, medians, gains, gates) on whole windows of
    the workload, one window per host core over disjoint windows (the C
    oracle releases the GIL), so a step does the same per-window work as a
    GPU step on a bounded sample of its windows."""
    from concurrent.futures import ThreadPoolExecutor
    ws, rank, _ = dist_env()
    if rank != 0:
        return None
    from oracle import oracle as O
    O.build_lib()
    w = wl.by_name(args.workload, seed=args.seed, steps=args.steps_override)
    cores = os.cpu_count() or 1
    nwin = max(1, min(cores, w.T // w.W))
    slices = [w.generate(t0=i * w.W, nsteps=min(w.W, w.T - i * w.W)) for i in range(nwin)]
    sw = wl.Workload(**{**w.__dict__, "T": w.W})

    def step():
        with ThreadPoolExecutor(nwin) as ex:
            list(ex.map(lambda x: oracle_step(O, sw, x), slices))

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    secs = time.perf_counter() - t0
    rec = sum(x.shape[0] for x in slices) * w.R * w.S
    value = rec * args.steps / secs
    sample = (f"each step: windows 0..{nwin - 1} of {w.name} ({nwin} whole windows of {w.W} steps, "
              f"{rec} records), one per host thread, C oracle")
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "int64",
        "data": "synthetic", "config": workload_config(w, args, ws),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": nwin, "kind": "oracle", "sample": sample,
                         "host_cpus": cores, "cpu_model": cpu_model()},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


CONFIG_NAMES = ["tiny", "ddp128", "fsdp1024", "accum8192"] + [f"sweep_R{R}_S{S}" for R in wl.SWEEP_R
                                                                for S in wl.SWEEP_S]
# a single window of few steps over many ranks (the per-window use of Sec. 3):
# fewer steps than SMs
FEW_STEP_NAMES = ["steps_T100_R8192_S8", "steps_T8_R8192_S8", "steps_T1_R8192_S8", "steps_T64_R65536_S8"]
# 1 GiB shapes outside the tiled streaming path (odd S with R*S not a multiple
# of 16; more than 16 stages): the generic kernels
GENERIC_NAMES = ["sweep_R1000_S5", "sweep_R512_S24"]
ORACLE_SAMPLE_RECORDS = 4_000_000  # per oracle thread, per configuration


def measure_config(name: str, sf, device, peak: float, steps: int, warmup: int, seed: int, oracle=None) -> dict:
    """Frontier pass (sf_frontier), aggregation pass (sf_window_aggregate) and
    whole step on one synthetic configuration, device-resident, CUDA events;
    with `oracle`, the CPU oracle on a bounded sample of the same workload,
    single-threaded and on all host cores."""
    if name.startswith("sweep_"):
        R, S = (int(x[1:]) for x in name.split("_")[1:])
        w = wl.sweep(R, S, seed=seed)
    elif name.startswith("steps_"):
        T, R, S = (int(x[1:]) for x in name.split("_")[1:])
        w = wl.sweep(R, S, seed=seed, steps=T)
    else:
        w = wl.by_name(name, seed=seed)
    host = torch.empty((w.T, w.R, w.S), dtype=torch.int64, pin_memory=True)
    w.fill(host.numpy().reshape(-1), threads=os.cpu_count() or 1)
    d = host.to(device)
    del host
    st = sf.new_status(device)
    e = lambda shape, dt: torch.empty(shape, dtype=dt, device=device)  # noqa: E731
    fr = (e((w.T, w.S), torch.int64), e((w.T, w.S), torch.int32), e((w.T,), torch.int64))
    frontier = lambda: sf.sf_frontier(d, a=fr[0], lead=fr[1], makespan=fr[2], status=st)  # noqa: E731
    pipe = Pipeline(sf, w, d)
    din = w.T * w.R * w.S * 8
    rec = {"config": name, "R": w.R, "S": w.S, "T": w.T, "W": w.W, "gbytes": round(din / 1e9, 3)}
    if din < L2_FLUSH_BYTES:
        # input smaller than twice the L2: every timed step after an L2 flush
        rec["l2"] = f"input < 2 x L2: {L2_FLUSH_BYTES >> 20} MB read before each step, events around each step"
        timed = lambda fn: timed_loop_flushed(fn, steps, warmup, device)  # noqa: E731
    else:
        rec["l2"] = "input > L2 on every pass; back-to-back steps queued ahead"
        timed = lambda fn: timed_loop(fn, steps, warmup, 1, device, True, ahead=True)  # noqa: E731
    f_secs = timed(frontier) / steps
    f_bytes = din + w.T * w.S * 12 + w.T * 8
    rec["frontier"] = {"ms": round(f_secs * 1e3, 4), "gbs": round(f_bytes / f_secs / 1e9, 1),
                       "frac": round(f_bytes / f_secs / 1e9 / peak, 4), "records_per_s": w.records / f_secs}
    a_secs = timed(pipe.aggregate) / steps
    a_bytes = pipe.algorithmic_bytes()["window_aggregate"]
    rec["aggregate"] = {"ms": round(a_secs * 1e3, 4), "gbs": round(a_bytes / a_secs / 1e9, 1),
                        "frac": round(a_bytes / a_secs / 1e9 / peak, 4)}
    s_secs = timed(pipe.step) / steps
    rec["step"] = {"ms": round(s_secs * 1e3, 4), "records_per_s": w.records / s_secs}
    torch.cuda.synchronize()
    rec["status"] = int(st.item()) | int(pipe.status.item())
    del d, pipe, fr
    torch.cuda.empty_cache()
    if oracle is not None:
        n = max(1, ORACLE_SAMPLE_RECORDS // (w.R * w.S))
        cores = os.cpu_count() or 1
        one = oracle_rate(oracle, w, n, 1)
        allc = oracle_rate(oracle, w, n, max(1, min(cores, w.T // n)))
        rec["oracle"] = {"records_per_s_1core": one["value"], "records_per_s_all_cores": allc["value"],
                         "cores": allc["cores"], "sample": allc["sample"] + " (single-core: the first slice)"}
        rec["gpu_over_oracle_all_cores"] = round(rec["step"]["records_per_s"] / allc["value"], 1)
    return rec


def run_configs(args):
    """Throughput of the frontier pass (sf_frontier), the aggregation pass
    (sf_window_aggregate) and the whole step on every synthetic configuration:
    the four workloads and the 1 GiB bandwidth sweep.  One GPU; one JSON line
    with a record per configuration."""
    device = torch.device("cuda", 0)
    torch.cuda.set_device(device)
    import __graft_entry__
    __graft_entry__.build()
    from paper_2606_06751_gb300 import stagefrontier as sf

    peak, peak_kind = peaks()
    names = CONFIG_NAMES + FEW_STEP_NAMES + GENERIC_NAMES
    if args.only:
        names = [n for n in names if n in args.only.split(",")]
    out = [measure_config(n, sf, device, peak, args.steps, args.warmup, args.seed) for n in names]
    return add_nominal({"metric": "per-configuration throughput (frontier pass, aggregation pass, whole step)",
                        "unit": "GB/s and records/s", "peak_gbs": peak, "peak_kind": peak_kind,
                        "peaks": peaks_record(peak, peak_kind), "steps": args.steps, "warmup": args.warmup,
                        "configs": out}, peak, peak_kind)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="accum8192")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--steps-override", type=int, default=None, help="shrink T (tests only)")
    ap.add_argument("--cpu-sample-windows", type=int, default=2)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true", help="skip the per-configuration block")
    ap.add_argument("--configs", action="store_true",
                    help="throughput on every synthetic configuration instead of the benchmark step")
    ap.add_argument("--only", default=None, help="with --configs: comma-separated configuration names")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.configs:
        line = run_configs(args)
    else:
        line = run_reference(args) if args.impl == "reference" else run_ours(args)
    if line is not None:
        print(json.dumps(line), flush=True)
    if torch.distributed.is_initialized():
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
