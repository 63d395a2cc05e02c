#!/usr/bin/env python
"""Benchmark of the H-Scale hot path on GB300 (one JSON line on rank 0).

A step is one pass of the whole hot path over one synthetic layer with its inputs
resident in HBM: the Hessian-diagonal pass over every calibration chunk
(h_j += sum_t x_tj^2, Sec. 3.2), the global scale + RTN codes (Eq. 7), and the
H-Scale window search fused with the final re-quantization and packing
(Algorithm 1).  Default workload: Llama-style 8B q_proj, W [4096, 4096] bf16,
262144 calibration tokens of width 4096 streamed in 8192-token chunks, window
k = +-4.

value      groups quantized per second by the whole step (all ranks), inputs in HBM
e2e        the same through the public API with host buffers: the step's X chunks
           and W copied from pinned host memory (chunk copies overlap the Hessian
           pass on a second stream) and the codes + nibbles copied back
roofline   the dominant kernel (the Hessian pass): algorithmic bytes per launch over
           its CUDA-event time, against the measured HBM copy bandwidth
cpu_baseline  the fp64 CPU oracle on a bounded sample of the same workload

Multi-GPU: every rank quantizes its own layer (independent problems, no data-path
collective): weak scaling.  ``--impl reference`` times the CPU oracle instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import sys
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2608_28113_gb300 import workloads as wl  # noqa: E402

METRIC = "scale-search groups/s and Hessian-diag GB/s on 1 GB300, % of roofline"
UNIT = "groups/s"
HBM_SPEC_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["hscale", "reference"], default="hscale")
    p.add_argument("--workload", default="llama8b-q_proj", choices=sorted(wl.WORKLOADS))
    p.add_argument("--k", type=int, default=None, help="window half-width (default: workload's)")
    p.add_argument("--tokens", type=int, default=None,
                   help="calibration tokens per step (default: the workload's; smaller for ncu captures)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    return p.parse_args()


# ------------------------------------------------------------------ distributed plumbing
class Dist:
    def __init__(self, gpus: int):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            backend = "nccl" if torch.cuda.is_available() else "gloo"
            dist.init_process_group(backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            if torch.cuda.is_available():
                self.pg.barrier(device_ids=[torch.cuda.current_device()])
            else:
                self.pg.barrier()

    def max(self, v: float) -> float:
        if not self.pg:
            return v
        t = torch.tensor([v], dtype=torch.float64,
                         device="cuda" if torch.cuda.is_available() else "cpu")
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ------------------------------------------------------------------ peaks and clocks
def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured", d
    except Exception:
        return FALLBACK_HBM_GBS, "fallback", {}


class ClockSampler:
    """SM clock and clock-event (throttle) reasons, read through NVML every ~2 ms on a
    background thread during the timed region (nothing is recorded without NVML)."""
    REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
               0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, device_index: int):
        self.device_index = device_index
        self.samples, self.max_mhz, self.reasons = [], None, set()
        self._nvml = None
        self._handle = None
        self._stop = False
        try:
            import ctypes
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                raise OSError("nvmlInit failed")
            h = ctypes.c_void_p()
            ok = False
            try:
                bus = torch.cuda.get_device_properties(device_index)
                bus_id = "%08x:%02x:%02x.0" % (bus.pci_domain_id, bus.pci_bus_id, bus.pci_device_id)
                ok = nv.nvmlDeviceGetHandleByPciBusId_v2(bus_id.encode(), ctypes.byref(h)) == 0
            except AttributeError:
                pass
            if not ok:
                vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")
                idx = int(vis[device_index]) if device_index < len(vis) and vis[device_index].strip().isdigit() else device_index
                if nv.nvmlDeviceGetHandleByIndex_v2(idx, ctypes.byref(h)) != 0:
                    raise OSError("no NVML handle")
            self._nvml, self._handle, self._ct = nv, h, ctypes
            v = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(v)) == 0:
                self.max_mhz = float(v.value)
        except Exception:
            self._nvml = None

    def _sample(self):
        ct, nv, h = self._ct, self._nvml, self._handle
        v = ct.c_uint()
        r = ct.c_ulonglong()
        if nv.nvmlDeviceGetClockInfo(h, 1, ct.byref(v)) == 0:
            self.samples.append(float(v.value))
        if nv.nvmlDeviceGetCurrentClocksEventReasons(h, ct.byref(r)) == 0:
            for bit, name in self.REASONS.items():
                if r.value & bit:
                    self.reasons.add(name)

    def _loop(self):
        while not self._stop:
            self._sample()
            time.sleep(0.002)

    def __enter__(self):
        if self._nvml is not None:
            import threading
            self._sample()
            self._thread = threading.Thread(target=self._loop, daemon=True)
            self._thread.start()
        return self

    def __exit__(self, *a):
        if self._nvml is not None:
            self._stop = True
            self._thread.join()
            self._sample()

    def summary(self):
        return {"sm_mhz": statistics.median(self.samples) if self.samples else None,
                "sm_max_mhz": self.max_mhz, "reasons": sorted(self.reasons),
                "samples": len(self.samples), "source": "nvml" if self._nvml else "none"}


def profiled_traffic(workload: str, chunk: int, n: int):
    """DRAM bytes per Hessian launch from the committed ncu summary, if the kernel's sources
    are unchanged since that capture and the launch shape matches; else None."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"hessian_colsumsq_{workload}.traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        h = hashlib.sha256()
        for src in d["kernel_sources"]:
            with open(os.path.join(ROOT, src), "rb") as f:
                h.update(f.read())
        if h.hexdigest() != d["kernel_sources_sha256"] or d["chunk_tokens"] != chunk or d["n"] != n:
            return None
        return int(d["dram_bytes_per_launch"])
    except Exception:
        return None


# ------------------------------------------------------------------ workload
class Layer:
    """Device-resident inputs and outputs of one layer of a workload."""

    def __init__(self, W: wl.Workload, rank: int, k: int, device, tokens=None):
        L = W.layers[0]
        self.W, self.k = W, k
        self.m, self.n = L.out_features, L.in_features
        self.chunk = W.chunk_tokens[self.n]
        self.nchunks = max(1, (tokens or W.tokens) // self.chunk)
        self.tokens = self.nchunks * self.chunk
        seed = W.seed + 7919 * rank
        self.seed = seed
        a = wl.channel_magnitudes(self.n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult,
                                  seed, device=device)
        self.x = torch.empty(self.tokens, self.n, dtype=torch.bfloat16, device=device)
        for c in range(self.nchunks):
            wl.activation_chunk(self.chunk, a, seed, c, out=self.x[c * self.chunk:(c + 1) * self.chunk])
        self.w = wl.weight(self.m, self.n, W.sigma_w, seed, device=device)
        self.groups = self.m * self.n // 16
        self.h = torch.zeros(self.n, dtype=torch.float32, device=device)
        self.sg = torch.empty(1, dtype=torch.float32, device=device)
        self.codes0 = torch.empty(self.m, self.n // 16, dtype=torch.uint8, device=device)
        self.codes = torch.empty_like(self.codes0)
        self.packed = torch.empty(self.m, self.n // 2, dtype=torch.uint8, device=device)


def hessian_phase(hs, L: Layer, x=None):
    """h = 0, then one hscale_hessian_diag_accumulate per calibration chunk."""
    x = L.x if x is None else x
    L.h.zero_()
    for c in range(L.nchunks):
        hs.hscale_hessian_diag_accumulate(x[c * L.chunk:(c + 1) * L.chunk], L.h)


def scale_phase(hs, L: Layer, w=None):
    """Global scale + RTN codes, then the H-Scale search with the final packing."""
    w = L.w if w is None else w
    hs.hscale_rtn_scales(w, L.sg, L.codes0, L.ws)
    hs.hscale_refine_scales(w, L.h, L.sg, L.codes0, L.k, L.k, L.codes, L.packed)


def run_step(hs, L: Layer, ev=None):
    """One eager pass of the hot path.  ev: optional 3 events (start, after h, end)."""
    if ev:
        ev[0].record()
    hessian_phase(hs, L)
    if ev:
        ev[1].record()
    scale_phase(hs, L)
    if ev:
        ev[2].record()


def capture_graphs(hs, L: Layer):
    """The step's launch sequence captured as two CUDA graphs (Hessian pass; scales)."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        run_step(hs, L)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    gh, gs = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
    with torch.cuda.graph(gh):
        hessian_phase(hs, L)
    with torch.cuda.graph(gs):
        scale_phase(hs, L)
    torch.cuda.synchronize()
    return gh, gs


KERNELS_PER_STEP_FIXED = 3  # amax, rtn codes, refine


# ------------------------------------------------------------------ CPU oracle baseline
def cpu_baseline(W: wl.Workload, k: int, budget_s: float = 12.0):
    """Time the fp64 oracle on a bounded sample of the workload and extrapolate the
    whole-step time: Hessian over sampled tokens, RTN over the whole W, search over
    sampled rows."""
    import oracle
    oracle.build()
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.set_threads(cores)
    L = W.layers[0]
    m, n = L.out_features, L.in_features
    a = wl.channel_magnitudes(n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult, W.seed)
    tok = min(W.chunk_tokens[n], 4096)
    xb = wl.bf16_bits(wl.activation_chunk(tok, a, W.seed, 0))
    wb = wl.bf16_bits(wl.weight(m, n, W.sigma_w, W.seed))
    h = np.zeros(n)
    t0 = time.perf_counter()
    reps = 0
    while True:
        oracle.hessian_accumulate(xb, h)
        reps += 1
        if time.perf_counter() - t0 > budget_s / 3:
            break
    t_h = (time.perf_counter() - t0) / (reps * tok * n)        # seconds per token*channel
    t0 = time.perf_counter()
    s_g, _ = oracle.global_scale(wb)
    oracle.rtn_codes(wb, s_g)
    t_rtn = time.perf_counter() - t0
    h32 = h.astype(np.float32)
    rows = max(8, min(m, 64))
    t0 = time.perf_counter()
    done = 0
    while True:
        r0 = (done * rows) % m
        oracle.refine(wb[r0:r0 + rows], h32, s_g, None, k, k)
        done += 1
        if time.perf_counter() - t0 > budget_s / 3:
            break
    t_g = (time.perf_counter() - t0) / (done * rows * n // 16)  # seconds per group
    groups = m * n // 16
    step = t_h * W.tokens * n + t_rtn + t_g * groups
    return {
        "value": groups / step, "unit": UNIT, "cores": cores, "kind": "oracle",
        "sample": (f"fp64 C oracle, {cores} threads: Hessian over {tok}x{n} tokens*channels "
                   f"x{reps}, global scale + RTN over the whole {m}x{n} W, search over "
                   f"{done}x{rows} rows (k={k}); step time extrapolated to {W.tokens} tokens "
                   f"and {groups} groups"),
        "seconds_per_step": step,
        "hessian_tokens_channels_per_s": 1.0 / t_h,
        "search_groups_per_s": 1.0 / t_g,
    }


def reference_arm(args, d: Dist):
    """--impl reference: the CPU oracle, as it stands, on the host cores."""
    if d.rank != 0:
        return
    W = wl.WORKLOADS[args.workload]
    k = args.k if args.k is not None else W.window[0]
    vals = []
    cb = None
    for i in range(args.warmup + args.steps):
        cb = cpu_baseline(W, k, budget_s=3.0)
        if i >= args.warmup:
            vals.append(cb["seconds_per_step"])
    L = W.layers[0]
    groups = L.out_features * L.in_features // 16
    sec = statistics.mean(vals)
    value = groups / sec
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": W.name, "m": L.out_features, "n": L.in_features,
                   "tokens": W.tokens, "k": k},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cb["cores"], "kind": "oracle",
                         "sample": cb["sample"]},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ GPU arm
def gpu_arm(args, d: Dist):
    import paper_2608_28113_gb300 as hs
    hs.load()
    torch.cuda.set_device(d.local)
    dev = torch.device("cuda", d.local)
    W = wl.WORKLOADS[args.workload]
    k = args.k if args.k is not None else W.window[0]
    L = Layer(W, d.rank, k, dev, tokens=args.tokens)
    L.ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()

    warm = max(args.warmup, 3)
    for _ in range(warm):
        run_step(hs, L)
    torch.cuda.synchronize()

    # eager launches (one API call per chunk), for reference
    ev_e = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    torch.cuda.synchronize()
    for s in range(args.steps):
        run_step(hs, L, ev=ev_e[s])
    torch.cuda.synchronize()
    ms_eager = sum(e[0].elapsed_time(e[2]) for e in ev_e) / args.steps

    # timed region: the same launches replayed from CUDA graphs
    gh, gs = capture_graphs(hs, L)
    for _ in range(warm):
        gh.replay()
        gs.replay()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    d.barrier()
    torch.cuda.synchronize()
    with ClockSampler(d.local) as clk:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for s in range(args.steps):
            evs[s][0].record()
            gh.replay()
            evs[s][1].record()
            gs.replay()
            evs[s][2].record()
        t1.record()
        torch.cuda.synchronize()
    d.barrier()
    ms_total = t0.elapsed_time(t1)
    ms_h = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    ms_sc = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps
    ms_step = d.max(ms_total / args.steps)
    value = L.groups * d.world / (ms_step * 1e-3)

    # per-kernel times of the scale phase (rtn_scales; refine) from an eager loop
    ev_k = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    for s in range(args.steps):
        hs.hscale_rtn_scales(L.w, L.sg, L.codes0, L.ws)
        ev_k[s][0].record()
        hs.hscale_rtn_scales(L.w, L.sg, L.codes0, L.ws)
        ev_k[s][1].record()
        hs.hscale_refine_scales(L.w, L.h, L.sg, L.codes0, L.k, L.k, L.codes, L.packed)
        ev_k[s][2].record()
    torch.cuda.synchronize()
    ms_rtn = sum(e[0].elapsed_time(e[1]) for e in ev_k) / args.steps
    ms_ref = sum(e[1].elapsed_time(e[2]) for e in ev_k) / args.steps

    # ---- roofline of the dominant kernel (the Hessian pass)
    hbm_peak, peak_kind, peaks = measured_peaks()
    h_bytes_launch = 2 * L.chunk * L.n + 8 * L.n          # X read + h read/write
    ms_h_launch = ms_h / L.nchunks
    h_gbs = h_bytes_launch / (ms_h_launch * 1e-3) / 1e9
    # ---- search roofline: max(42 B/group over HBM, 80*C ops/group over the FP32 peak)
    props = torch.cuda.get_device_properties(dev)
    sm_max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_peak = props.multi_processor_count * 128 * sm_max_mhz * 1e6
    C = 2 * k + 1
    t_bytes = 42 * L.groups / (hbm_peak * 1e9)
    t_ops = 80 * C * L.groups / fp32_peak
    t_search_roof = max(t_bytes, t_ops)
    search_frac = t_search_roof / (ms_ref * 1e-3)

    # ---- end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        e2e = e2e_leg(hs, L, args)

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": d.world, "steps": args.steps,
        "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "input_dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": W.name, "m": L.m, "n": L.n, "tokens": L.tokens,
                   "chunk_tokens": L.chunk, "k": k, "groups": L.groups,
                   "l2": f"inputs larger than L2: {L.tokens * L.n * 2 / 1e9:.2f} GB of X streamed per step",
                   "parallelism": f"independent layer per GPU x{d.world}"},
        "roofline": {"bound": "hbm", "kernel": "hessian_colsumsq", "achieved": h_gbs,
                     "peak": hbm_peak, "unit": "GB/s", "frac": h_gbs / hbm_peak,
                     "peak_kind": f"{peak_kind} HBM copy bandwidth",
                     "frac_of_8TBs_spec": h_gbs / HBM_SPEC_GBS,
                     "traffic": profiled_traffic(W.name, L.chunk, L.n),
                     "bytes_per_launch": h_bytes_launch, "ms_per_launch": ms_h_launch},
        "phases_ms": {"hessian": ms_h, "scales": ms_sc, "rtn_scales": ms_rtn, "refine": ms_ref},
        "ms_per_step_eager": ms_eager,
        "timed_launch": "CUDA graphs of the step's API calls (Hessian pass; scales)",
        "hessian": {"gbs": h_gbs, "tokens_channels_per_s": L.chunk * L.n / (ms_h_launch * 1e-3),
                    "frac_of_measured_hbm": h_gbs / hbm_peak, "frac_of_8TBs": h_gbs / HBM_SPEC_GBS},
        "search": {"groups_per_s": L.groups / (ms_ref * 1e-3), "candidates": C,
                   "bound": "alu" if t_ops > t_bytes else "hbm",
                   "roofline_s": t_search_roof, "frac": search_frac,
                   "fp32_peak_ops": fp32_peak, "sm_count": props.multi_processor_count,
                   "clock_mhz_for_peak": sm_max_mhz},
        "seconds_per_layer": ms_step * 1e-3,
        "clocks": clk.summary(),
        "gpu_launches": args.steps * (L.nchunks + KERNELS_PER_STEP_FIXED),
    }
    if e2e:
        line["e2e"] = e2e
    if d.rank == 0 and d.world == 1 and not args.no_cpu_baseline:
        cb = cpu_baseline(W, k)
        line["cpu_baseline"] = {k2: cb[k2] for k2 in ("value", "unit", "cores", "kind", "sample")}
    if d.rank == 0:
        print(json.dumps(line), flush=True)


def e2e_leg(hs, L: Layer, args):
    """Whole step through the public API with host buffers: X chunks and W copied from
    pinned host memory inside the timed region (chunk copies on a copy stream overlap
    the Hessian pass), codes and nibbles copied back."""
    dev = L.x.device
    x_host = torch.empty(L.x.shape, dtype=L.x.dtype, pin_memory=True)
    x_host.copy_(L.x)
    w_host = torch.empty(L.w.shape, dtype=L.w.dtype, pin_memory=True)
    w_host.copy_(L.w)
    codes_host = torch.empty(L.codes.shape, dtype=torch.uint8, pin_memory=True)
    packed_host = torch.empty(L.packed.shape, dtype=torch.uint8, pin_memory=True)
    nbuf = 3
    xbuf = [torch.empty(L.chunk, L.n, dtype=torch.bfloat16, device=dev) for _ in range(nbuf)]
    wdev = torch.empty_like(L.w)
    copy = torch.cuda.Stream(device=dev)
    comp = torch.cuda.current_stream(dev)

    def step():
        done = [torch.cuda.Event() for _ in range(nbuf)]
        ready = [torch.cuda.Event() for _ in range(L.nchunks)]
        L.h.zero_()
        for c in range(L.nchunks):
            b = c % nbuf
            with torch.cuda.stream(copy):
                if c >= nbuf:
                    copy.wait_event(done[b])
                xbuf[b].copy_(x_host[c * L.chunk:(c + 1) * L.chunk], non_blocking=True)
                ready[c].record(copy)
            comp.wait_event(ready[c])
            hs.hscale_hessian_diag_accumulate(xbuf[b], L.h)
            done[b].record(comp)
        with torch.cuda.stream(copy):
            wdev.copy_(w_host, non_blocking=True)
            wr = torch.cuda.Event()
            wr.record(copy)
        comp.wait_event(wr)
        hs.hscale_rtn_scales(wdev, L.sg, L.codes0, L.ws)
        hs.hscale_refine_scales(wdev, L.h, L.sg, L.codes0, L.k, L.k, L.codes, L.packed)
        codes_host.copy_(L.codes, non_blocking=True)
        packed_host.copy_(L.packed, non_blocking=True)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 10))
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record()
    for _ in range(reps):
        step()
    t1.record()
    torch.cuda.synchronize()
    ms = t0.elapsed_time(t1) / reps
    h2d = L.tokens * L.n * 2 + L.m * L.n * 2
    d2h = L.codes.numel() + L.packed.numel()
    del x_host
    return {"value": L.groups / (ms * 1e-3), "unit": UNIT, "ms_per_step": ms,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}


def main():
    args = parse()
    d = Dist(args.gpus)
    try:
        if args.impl == "reference":
            reference_arm(args, d)
        else:
            if not torch.cuda.is_available():
                raise SystemExit("bench.py needs a CUDA device")
            gpu_arm(args, d)
    finally:
        d.close()


if __name__ == "__main__":
    main()
