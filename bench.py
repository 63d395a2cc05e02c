#!/usr/bin/env python
"""Benchmark of the H-Scale hot path on GB300 (one JSON line on rank 0).

A step is one pass of the whole hot path over one synthetic layer with its inputs
resident in HBM: for every input space the Hessian-diagonal pass over all calibration
chunks (h_j += sum_t x_tj^2, Sec. 3.2), and for every weight matrix the global scale +
RTN codes (Eq. 7) and the H-Scale window search fused with the final re-quantization and
packing (Algorithm 1).  Default workload: Llama-style 8B q_proj, W [4096, 4096] bf16,
262144 calibration tokens of width 4096 streamed in 8192-token chunks, window k = +-4.
Other workloads: the full 8B decoder layer (per-layer and per-model seconds), the MLP
down_proj, and the 70B MLP block with its window sweep.  The timed steps replay CUDA
graphs on three streams; steps with several input spaces, or whose searches outweigh
their Hessian passes, are pipelined (a step's last searches alongside the next step's
first Hessian pass, on alternating buffer sets).

value      groups quantized per second by the whole step (all ranks), inputs in HBM
e2e        the same through the public API with host buffers: the X chunks and W copied
           from pinned host memory (chunk copies overlap the Hessian pass on a second
           stream) and the codes + nibbles copied back
roofline   the dominant kernel (the Hessian pass): algorithmic bytes per launch over its
           CUDA-event time, against the measured HBM copy bandwidth
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
    p.add_argument("--workload", default="llama8b-decoder", choices=sorted(wl.WORKLOADS),
                   help="the step's workload (default: one layer of the full 8B decoder, the largest "
                        "single-GPU configuration; per-model time = 32 layers)")
    p.add_argument("--extra-workload", default="llama70b-mlp", choices=["none"] + sorted(wl.WORKLOADS),
                   help="a second workload measured in the same process and reported under its own key "
                        "(default: the 70B MLP block with its window sweep k = 1, 2, 4, 8, 16)")
    p.add_argument("--k", type=int, default=None, help="symmetric window half-width (default: workload's first)")
    p.add_argument("--window", default=None,
                   help="asymmetric window 'D,U' (codes c0-D .. c0+U); e.g. 9,6 is the paper's K = 16 default")
    p.add_argument("--tokens", type=int, default=None,
                   help="calibration tokens per input space (default: the workload's; smaller for ncu captures)")
    p.add_argument("--init", choices=["rtn", "4over6", "4over6-2pass"], default="rtn",
                   help="initial codes of the search: max-abs RTN (Eq. 7), or 4over6 (Algorithm 2) "
                        "decided inside the search (one pass) or by a separate codes pass")
    p.add_argument("--col-block", type=int, default=0,
                   help="channels per column block of the step: each block's Hessian pass over every "
                        "token, then that block's searches alongside the next block's Hessian pass "
                        "(a multiple of 64).  0 (default): whole input spaces, Hessian pass in token "
                        "chunks; on q_proj blocks of 512-2048 channels make the Hessian pass 5-38 %% "
                        "slower (each launch reads a fraction of every row) and the step slower")
    p.add_argument("--overlap-ctas", type=int, default=-1,
                   help="resident search CTAs per SM while the next input space's Hessian pass "
                        "runs alongside (0: run every search after the last Hessian pass; -1, the "
                        "default: when the step's estimated search time exceeds its Hessian time, 7 "
                        "(every CTA the search kernel keeps resident); else 4)")
    p.add_argument("--search-schedule", choices=["auto", "shared", "static"], default="auto",
                   help="the search's unit schedule: 'shared' passes hscale_refine_scales_ws a workspace "
                        "(units shared out at run time in long searches), 'static' passes none; 'auto' "
                        "shares except in searches that fill the SMs beside a Hessian pass")
    p.add_argument("--weight-pass", choices=["early", "with-search"], default="early",
                   help="where the graphs put each matrix's weight-only calls (s_g): 'early' on a side "
                        "stream alongside the first Hessian pass; 'with-search' on the search stream "
                        "right before the matrix's search (its W may still be in L2)")
    p.add_argument("--pipeline", choices=["auto", "on", "off"], default="auto",
                   help="run each step's last searches alongside the next step's first Hessian pass "
                        "(h, s_g and initial codes double-buffered).  auto (default) and on: pipelined "
                        "(decoder layer -4 %%, 70B MLP block -9 %%, q_proj -8 %% per step); off: each "
                        "step ends when its last searches do")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-baseline", choices=["full", "sample"], default="full",
                   help="full (default): the oracle over the step's whole layer on all host cores, "
                        "verified against the GPU outputs; sample: a bounded sample extrapolated")
    p.add_argument("--no-output-error", action="store_true",
                   help="skip the tensor-core layer-output error evaluation")
    p.add_argument("--no-gptq", action="store_true",
                   help="skip the GPTQ + H-Scale (Algorithm 3) evaluation")
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
            from datetime import timedelta
            backend = "nccl" if torch.cuda.is_available() else "gloo"
            # a rank that dies or never arrives makes the others' next collective fail
            # after this long instead of hanging
            timeout = timedelta(seconds=float(os.environ.get("HSCALE_PG_TIMEOUT_S", "600")))
            dist.init_process_group(backend, timeout=timeout)
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


def step_traffic(work) -> float | None:
    """DRAM bytes per Hessian launch of the step (the mean over its launches), from the
    committed ncu summaries (profiles/hessian_colsumsq_*.traffic.json): one figure per
    launch shape (chunk tokens, channels), taken from any summary whose kernel sources hash
    to the current ones.  None when no such summary covers every launch shape of the step."""
    import glob
    import hashlib
    per_shape = {}
    for path in sorted(glob.glob(os.path.join(ROOT, "profiles", "hessian_colsumsq_*.traffic.json"))):
        try:
            with open(path) as f:
                d = json.load(f)
            h = hashlib.sha256()
            for src in d["kernel_sources"]:
                with open(os.path.join(ROOT, src), "rb") as f:
                    h.update(f.read())
            if h.hexdigest() != d["kernel_sources_sha256"]:
                continue
            for e in d["shapes"]:
                per_shape[(int(e["chunk_tokens"]), int(e["n"]))] = float(e["dram_bytes_per_launch"])
        except Exception:
            continue
    total, launches = 0.0, 0
    for S, c0, c1 in work.pieces:
        for t0, t1 in hessian_calls(S, c0, c1):
            key = (t1 - t0, c1 - c0)
            if key not in per_shape:
                return None
            total += per_shape[key]
            launches += 1
    return total / launches if launches else None


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


# ------------------------------------------------------------------ workload
class Space:
    """One input space: resident calibration activations X [tokens, n] and its h."""

    def __init__(self, W: wl.Workload, name: str, n: int, seed: int, device, tokens=None):
        self.name, self.n = name, n
        self.chunk = W.chunk_tokens[n]
        self.nchunks = max(1, (tokens or W.tokens) // self.chunk)
        self.tokens = self.nchunks * self.chunk
        a = wl.channel_magnitudes(n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult,
                                  wl.chunk_seed(seed, name, 0) & 0xFFFFFFFF, device=device)
        self.x = torch.empty(self.tokens, n, dtype=torch.bfloat16, device=device)
        for c in range(self.nchunks):
            wl.activation_chunk(self.chunk, a, wl.chunk_seed(seed, name, 1) & 0xFFFFFFFF, c,
                                out=self.x[c * self.chunk:(c + 1) * self.chunk])
        self.h = torch.zeros(n, dtype=torch.float32, device=device)


class Matrix:
    """One weight matrix with its outputs; uses the h of its input space."""

    def __init__(self, W: wl.Workload, L: wl.LayerShape, space: Space, seed: int, device):
        self.name, self.m, self.n, self.space = L.name, L.out_features, L.in_features, space
        self.w = wl.weight(self.m, self.n, W.sigma_w, wl.chunk_seed(seed, L.name, 0) & 0xFFFFFFFF,
                           device=device)
        self.groups = self.m * self.n // 16
        self.sg = torch.empty(1, dtype=torch.float32, device=device)
        self.codes0 = torch.empty(self.m, self.n // 16, dtype=torch.uint8, device=device)
        self.codes = torch.empty_like(self.codes0)
        self.packed = torch.empty(self.m, self.n // 2, dtype=torch.uint8, device=device)
        # the search's work-sharing counter (hscale_refine_workspace_bytes(); the calls of one
        # matrix never overlap on the GPU)
        self.sched = torch.zeros(16, dtype=torch.uint8, device=device)


def column_blocks(S: Space, col_block: int):
    """Column blocks [c0, c1) of an input space: the whole width when col_block is 0 or
    not smaller than n."""
    if col_block <= 0 or col_block >= S.n:
        return [(0, S.n)]
    return [(c0, min(S.n, c0 + col_block)) for c0 in range(0, S.n, col_block)]


def hessian_calls(S: Space, c0: int, c1: int):
    """Token ranges (t0, t1) of the Hessian calls over the channels [c0, c1): the space's
    chunks for the whole width, else launches of about a chunk's bytes."""
    rows = S.chunk if c1 - c0 == S.n else max(S.chunk, S.chunk * S.n // (c1 - c0))
    return [(t0, min(S.tokens, t0 + rows)) for t0 in range(0, S.tokens, rows)]


class Work:
    """Device-resident inputs and outputs of one layer of a workload."""

    def __init__(self, W: wl.Workload, rank: int, win, device, tokens=None, init="rtn", col_block=0):
        if col_block % 64:
            raise SystemExit("--col-block must be a multiple of 64")
        self.W, self.win, self.init, self.col_block = W, tuple(win), init, col_block
        self.seed = W.layer_seed(0) + 7919 * rank
        self.spaces = {name: Space(W, name, n, self.seed, device, tokens) for name, n in W.input_spaces()}
        self.mats = [Matrix(W, L, self.spaces[L.input_space], self.seed, device) for L in W.layers]
        self.groups = sum(M.groups for M in self.mats)
        # pieces of the step in order: (space, c0, c1), spaces in flow-shop order
        self.pieces = [(S, c0, c1) for S in self.space_order() for c0, c1 in column_blocks(S, col_block)]
        calls = [(c1 - c0, t1 - t0) for S, c0, c1 in self.pieces for t0, t1 in hessian_calls(S, c0, c1)]
        self.h_bytes = sum(2 * rows * width + 8 * width for width, rows in calls)
        self.h_launches = len(calls)
        self.ws = None
        self.search_schedule = "auto"
        self.weight_pass = "early"

    def stage_estimates(self):
        """(name, Hessian seconds, search seconds) per input space, from nominal rates
        (6.6 TB/s; 0.45 of 40 T lane operations per second); only their ratios matter."""
        cands = self.win[0] + self.win[1] + 1
        jobs = []
        for S in self.spaces.values():
            a = 2.0 * S.tokens * S.n / 6.6e12
            b = sum(M.groups for M in self.mats if M.space is S) * 80.0 * cands / (0.45 * 40.3e12)
            jobs.append((S.name, a, b))
        return jobs

    def search_bound(self) -> bool:
        """Do the step's searches take longer (estimated) than its Hessian passes?"""
        jobs = self.stage_estimates()
        return sum(j[2] for j in jobs) > sum(j[1] for j in jobs)

    def pipelined(self, requested: str) -> bool:
        """Whether consecutive steps overlap: unless asked not to.  With the Hessian pass's
        squares on the tensor cores it shares its SMs with the searches well enough that
        overlapping pays on every workload measured (1 GB300): decoder layer 1.217 against
        1.271 ms per step, 70B MLP block 1.866 against 2.057 ms, q_proj 0.318 against
        0.345 ms."""
        return requested != "off"

    def overlap_ctas(self, requested: int, pipelined: bool) -> int:
        """Search CTAs per SM alongside a Hessian pass: the requested number, or by default
        4 when the Hessian passes outweigh the searches (decoder layer, pipelined: 1.217 ms,
        against 1.252 at 3 and 1.224 at 5; q_proj 0.318 ms).  When the searches outweigh
        them they take 7, every CTA the search kernel keeps resident (70B MLP block: 1.866 ms
        pipelined, against 1.995 at 6 and 2.089 at 5; 2.057 ms at 7 without pipelining,
        2.084 at 5).  The launcher clamps a larger number to the kernel's occupancy."""
        if requested >= 0:
            return requested
        return 7 if self.search_bound() else 4

    def space_order(self):
        """The input spaces in the order the step takes them.  Each space is a two-stage
        job: its Hessian pass (HBM-bound, about 2 bytes per token and channel) and then the
        searches of its matrices (ALU-bound, about 80 operations per group and candidate);
        the searches of one space run alongside the Hessian passes of the next, so
        Johnson's rule on the estimated stage times keeps both streams busy."""
        return [self.spaces[name] for name in johnson_order(self.stage_estimates())]


def johnson_order(jobs):
    """Order of two-stage jobs (name, a, b) -- stage 1 (time a) before stage 2 (time b), one
    machine per stage -- that minimises the makespan (Johnson's rule): jobs with a <= b
    first, by increasing a; then the others, by decreasing b."""
    first = sorted((j for j in jobs if j[1] <= j[2]), key=lambda j: j[1])
    last = sorted((j for j in jobs if j[1] > j[2]), key=lambda j: -j[2])
    return [j[0] for j in first + last]


def hessian_block(hs, S: Space, c0: int, c1: int):
    """h[c0:c1] = 0, then the Hessian calls over every token of the channels [c0, c1)."""
    h = S.h[c0:c1]
    h.zero_()
    for t0, t1 in hessian_calls(S, c0, c1):
        # X is resident and complete before the step starts: the chunk kernels may overlap
        hs.hscale_hessian_diag_accumulate_ex(S.x[t0:t1, c0:c1], h, hs.HSCALE_HESSIAN_X_READY)


def refine_block(hs, work: Work, M, c0: int, c1: int, down, up, ctas_per_sm=0):
    """The search of the columns [c0, c1) of one matrix, on 2-D views of W and its outputs."""
    if (c0, c1) == (0, M.n):
        return refine(hs, work, M, down, up, ctas_per_sm=ctas_per_sm)
    g0, g1 = c0 // 16, c1 // 16
    init = M.codes0[:, g0:g1] if work.init == "4over6-2pass" else None
    hs.hscale_refine_scales_strided(M.w[:, c0:c1], M.space.h[c0:c1], M.sg, init, work.init == "4over6", down, up,
                                    M.codes[:, g0:g1], M.packed[:, c0 // 2:c1 // 2], ctas_per_sm)


def init_codes(hs, work: Work, M, w=None):
    """The weight-only part of one matrix: the global scale s_g, and with the two-pass
    4over6 init Algorithm 2's codes.  With RTN or one-pass 4over6 init the search decides
    the initial codes itself, which saves a pass over W."""
    w = M.w if w is None else w
    hs.hscale_rtn_scales(w, M.sg, None, work.ws)
    if work.init == "4over6-2pass":
        hs.hscale_fourover6_codes(w, M.sg, M.codes0)


def init_phase(hs, work: Work, ws=None):
    for M in work.mats:
        init_codes(hs, work, M, None if ws is None else ws[M.name])


def refine(hs, work: Work, M, down, up, w=None, ctas_per_sm=0):
    """The H-Scale search with packing of one matrix over the window (down, up)."""
    w = M.w if w is None else w
    init = M.codes0 if work.init == "4over6-2pass" else None
    hs.hscale_refine_scales_ws(w, M.space.h, M.sg, init, int(work.init == "4over6"), down, up, M.codes, M.packed,
                               ctas_per_sm, M.sched if shares(work, ctas_per_sm) else None)


def shares(work: Work, ctas_per_sm: int) -> bool:
    """Whether a search call gets the work-sharing workspace.  With 'auto' every call does
    except one that fills the SMs (7 CTAs each) beside a Hessian pass: a static deal lets
    its first CTAs finish midway and make room for the Hessian pass's CTAs, while shared
    units keep every CTA resident to the end."""
    if work.search_schedule == "auto":
        return not 7 <= ctas_per_sm
    return work.search_schedule == "shared"


def refine_phase(hs, work: Work, win=None, ws=None):
    down, up = work.win if win is None else win
    for M in work.mats:
        refine(hs, work, M, down, up, None if ws is None else ws[M.name])


def scale_phase(hs, work: Work, win=None, ws=None):
    """For every matrix: the weight-only part, then the search."""
    init_phase(hs, work, ws)
    refine_phase(hs, work, win, ws)


def run_step(hs, work: Work):
    """One eager pass of the hot path on the current stream, piece by piece."""
    init_phase(hs, work)
    down, up = work.win
    for S, c0, c1 in work.pieces:
        hessian_block(hs, S, c0, c1)
        for M in work.mats:
            if M.space is S:
                refine_block(hs, work, M, c0, c1, down, up)


class StepGraphs:
    """The step's launches as CUDA graphs on three streams.  The step is a sequence of
    pieces: a column block [c0, c1) of one input space (a whole space when the step is
    not blocked).

    main:   the Hessian pass of each piece in turn (HBM-bound);
    side:   the weight-only calls of every matrix (s_g, 4over6 codes), alongside;
    search: the searches of a piece (the piece's columns of every matrix of its space;
            ALU-bound), started as soon as the piece's h is complete and the weight-only
            calls are done, so that they run alongside the next piece's Hessian pass.
            Those searches keep at most `overlap_ctas` CTAs resident per SM, which leaves
            registers for the Hessian CTAs.  overlap_ctas = 0 runs every search after the
            last Hessian pass instead.

    pipelined (when asked for and overlap_ctas > 0): consecutive steps overlap as well, so
    the last piece's searches run alongside the next step's first Hessian pass.  The
    buffers that one step's streams hand to each other -- h of every input space; s_g
    and the two-pass 4over6 codes of every matrix -- come in two sets, taken by
    alternate steps, and a step starts its Hessian passes and weight-only calls only
    once the searches of the step before the previous one, which read the same set, are
    done.  Without pipelining the last piece's searches fill the GPU and the step ends
    when they do."""

    def __init__(self, hs, work: Work, overlap_ctas: int, pipeline: bool = True):
        self.work, self.overlap = work, overlap_ctas > 0
        self.pipeline = pipeline and self.overlap
        spaces = list(work.spaces.values())
        self.sets = [({S.name: S.h for S in spaces}, {M.name: (M.sg, M.codes0) for M in work.mats})]
        if self.pipeline:
            self.sets.append(({S.name: torch.zeros_like(S.h) for S in spaces},
                              {M.name: (torch.empty_like(M.sg), torch.empty_like(M.codes0))
                               for M in work.mats}))
        down, up = work.win
        self.gh, self.gr, self.gi = [], [], []
        for p in range(len(self.sets)):
            self.bind(p)
            warm = torch.cuda.Stream()
            warm.wait_stream(torch.cuda.current_stream())
            with torch.cuda.stream(warm):
                run_step(hs, work)
            torch.cuda.current_stream().wait_stream(warm)
            torch.cuda.synchronize()
            gh, gr = [], []
            for i, (S, c0, c1) in enumerate(work.pieces):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    hessian_block(hs, S, c0, c1)
                gh.append(g)
                alongside = self.overlap and (self.pipeline or i + 1 < len(work.pieces))
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g):
                    for M in work.mats:
                        if M.space is S:
                            if work.weight_pass == "with-search" and c0 == 0:
                                init_codes(hs, work, M)
                            refine_block(hs, work, M, c0, c1, down, up,
                                         ctas_per_sm=overlap_ctas if alongside else 0)
                gr.append(g)
            gi = None
            if work.weight_pass == "early":
                gi = torch.cuda.CUDAGraph()
                with torch.cuda.graph(gi):
                    init_phase(hs, work)
            self.gh.append(gh)
            self.gr.append(gr)
            self.gi.append(gi)
        self.bind(0)
        torch.cuda.synchronize()
        self.side, self.search = torch.cuda.Stream(), torch.cuda.Stream()
        self.ev_init = torch.cuda.Event()
        self.ev_h = [torch.cuda.Event() for _ in work.pieces]
        self.done = [torch.cuda.Event() for _ in self.sets]
        self.used = [False for _ in self.sets]
        self.k = 0

    def bind(self, p: int):
        """Points the work's spaces and matrices at buffer set p."""
        hset, mset = self.sets[p]
        for S in self.work.spaces.values():
            S.h = hset[S.name]
        for M in self.work.mats:
            M.sg, M.codes0 = mset[M.name]

    def replay(self, ev=None):
        """One step.  ev: optional (start, after the last Hessian pass, end of the step's
        searches) timing events; the first two are recorded on the current stream, which
        runs the Hessian passes, the last on the search stream when pipelined.  A
        pipelined step may still be running when this returns: drain() joins it."""
        main = torch.cuda.current_stream()
        p = self.k % len(self.sets)
        self.k += 1
        if ev:
            ev[0].record()
        if self.pipeline and self.used[p]:
            main.wait_event(self.done[p])
        self.side.wait_stream(main)
        self.search.wait_stream(main)
        if self.gi[p] is not None:
            with torch.cuda.stream(self.side):
                self.gi[p].replay()
                self.ev_init.record(self.side)
            self.search.wait_event(self.ev_init)
        for i, g in enumerate(self.gh[p]):
            g.replay()
            self.ev_h[i].record(main)
            if self.overlap:
                self.search.wait_event(self.ev_h[i])
                with torch.cuda.stream(self.search):
                    self.gr[p][i].replay()
        if ev:
            ev[1].record()
        if not self.overlap:
            self.search.wait_stream(main)
            with torch.cuda.stream(self.search):
                for g in self.gr[p]:
                    g.replay()
        if self.pipeline:
            self.done[p].record(self.search)
            self.used[p] = True
            if ev:
                ev[2].record(self.search)
        else:
            self.drain()
            if ev:
                ev[2].record()

    def drain(self):
        """Joins every stream of the steps replayed so far into the current stream."""
        main = torch.cuda.current_stream()
        main.wait_stream(self.search)
        main.wait_stream(self.side)


# algorithmic bytes per group of the search: W 32, nibbles 8, code out 1, code in 1 (none
# when the search decides the initial codes itself)
SEARCH_BYTES = {"rtn": 41, "4over6": 41, "4over6-2pass": 42}
# algorithmic bytes per group of the weight-only calls: W 32 for the global amax, and with
# the two-pass 4over6 init W 32 again and the code written 1
WEIGHT_BYTES = {"rtn": 32, "4over6": 32, "4over6-2pass": 65}


def step_hbm(work, ms_step: float, hbm_peak: float, peak_kind: str) -> dict:
    """The whole step against HBM: every byte the step has to move (X once for the Hessian
    passes, W for the global amax and again in the search, the codes and nibbles written),
    over the step's time, against the copy bandwidth."""
    b = work.h_bytes + (WEIGHT_BYTES[work.init] + SEARCH_BYTES[work.init]) * work.groups
    gbs = b / (ms_step * 1e-3) / 1e9
    return {"bytes": b, "achieved": gbs, "peak": hbm_peak, "unit": "GB/s", "frac": gbs / hbm_peak,
            "peak_kind": f"{peak_kind} HBM copy bandwidth",
            "note": "X once, W twice (global amax, search), codes and nibbles out, over the whole step"}


def kernels_per_matrix(work: Work) -> int:
    """Library kernels per matrix and step: amax and s_g (hscale_rtn_scales), the 4over6
    codes with the two-pass init, the search."""
    return 4 if work.init == "4over6-2pass" else 3


# the search kernels: one CTA per SM with a shared-memory queue (a matrix alone on the GPU),
# the global work counter (long searches), the static deal (tiny searches)
SEARCH_KERNELS = "refine_sm_kernel|refine_shared_kernel|refine_linear_kernel"


def timed(fn, reps, flush=None):
    """Average CUDA-event time (ms) of fn over reps calls on the current stream, after one
    untimed call (library loading, handle creation and first-use costs stay out).  With
    `flush` (two device buffers, each larger than L2), each call is timed on its own after
    the first buffer is rewritten and the second read, outside the timed window, so inputs
    smaller than L2 (a weight matrix) are read from HBM every time, and the flush's dirty
    lines have been written back before the call starts.  The start event follows a short
    device-side spin (about 50 us), queued before the host makes the call, so the window
    holds the call's kernels and not the host's time to enqueue them."""
    fn()
    if flush is not None:
        total = 0.0
        for _ in range(reps):
            flush[0].fill_(1.0)
            flush[1].sum()
            torch.cuda.synchronize()
            torch.cuda._sleep(SPIN_CYCLES)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            fn()
            e1.record()
            torch.cuda.synchronize()
            total += e0.elapsed_time(e1)
        return total / reps
    torch.cuda.synchronize()
    torch.cuda._sleep(SPIN_CYCLES)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        fn()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


# device-side spin before a timed window: ~50 us at 2 GHz, longer than one host call
SPIN_CYCLES = 100_000


def timed_graph(fn, reps):
    """Average time (ms) of fn's work over reps replays of one CUDA graph that captured it
    (after one untimed eager call and one untimed replay).  For library calls made of many
    dependent launches, whose eager form waits on the host's launch latency at every step."""
    fn()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        fn()
    g.replay()
    torch.cuda.synchronize()
    torch.cuda._sleep(SPIN_CYCLES)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(reps):
        g.replay()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / reps


# ------------------------------------------------------------------ CPU oracle baseline
def window_of(args, W: wl.Workload):
    """(down, up) of the run: --window D,U, else --k, else the workload's first k."""
    if args.window:
        d, u = (int(v) for v in args.window.split(","))
        return (d, u)
    k = args.k if args.k is not None else W.window[0]
    return (k, k)


def _oracle_step(W: wl.Workload, win, budget_s: float, init: str, threads: int):
    """Whole-step time of the fp64 oracle with `threads` threads, extrapolated from a
    bounded sample: Hessian over sampled tokens of every input space, global scale +
    initial codes (RTN or 4over6) over every matrix, search over sampled rows of every
    matrix.  Returns (seconds per step, groups, samples, token-channels)."""
    import oracle
    oracle.set_threads(threads)
    per_part = budget_s / (len(W.input_spaces()) + len(W.layers))
    step = 0.0
    groups = 0
    h_tc = 0
    samples = []
    hs_of = {}
    for name, n in W.input_spaces():
        a = wl.channel_magnitudes(n, W.sigma_a, W.outlier_channels, W.outlier_channel_mult, W.seed)
        tok = min(W.chunk_tokens[n], 4096)
        xb = wl.bf16_bits(wl.activation_chunk(tok, a, W.seed, 0))
        h = np.zeros(n)
        t0 = time.perf_counter()
        reps = 0
        while True:
            oracle.hessian_accumulate(xb, h)
            reps += 1
            if time.perf_counter() - t0 > per_part:
                break
        t_tc = (time.perf_counter() - t0) / (reps * tok * n)
        step += t_tc * W.tokens * n
        h_tc += W.tokens * n
        hs_of[name] = (h / reps * (W.tokens / tok)).astype(np.float32)
        samples.append(f"Hessian {name}: {reps} passes over one {tok}-token x {n}-channel chunk")
    t_rtn_total = 0.0
    for L in W.layers:
        m, n = L.out_features, L.in_features
        wb = wl.bf16_bits(wl.weight(m, n, W.sigma_w, W.seed))
        t0 = time.perf_counter()
        s_g, _ = oracle.global_scale(wb)
        c0 = oracle.fourover6_codes(wb, s_g)[0] if init.startswith("4over6") else oracle.rtn_codes(wb, s_g)
        t_rtn_total += time.perf_counter() - t0
        rows = max(8, min(m, 64))
        t0 = time.perf_counter()
        done = 0
        while True:
            r0 = (done * rows) % m
            oracle.refine(wb[r0:r0 + rows], hs_of[L.input_space], s_g, c0[r0:r0 + rows], win[0], win[1])
            done += 1
            if time.perf_counter() - t0 > per_part:
                break
        t_g = (time.perf_counter() - t0) / (done * rows * n // 16)
        G = m * n // 16
        step += t_g * G
        groups += G
        samples.append(f"search {L.name}: {done} batches of {rows} rows")
    step += t_rtn_total
    return step, groups, samples, h_tc


def cpu_baseline(W: wl.Workload, win, budget_s: float = 12.0, init: str = "rtn"):
    """The fp64 oracle timed on the host's cores (all of them, and one thread on a shorter
    sample), extrapolated to the whole step from a bounded sample."""
    import oracle
    oracle.build()
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    step, groups, samples, h_tc = _oracle_step(W, win, budget_s, init, cores)
    step1, _, samples1, _ = _oracle_step(W, win, budget_s / 3, init, 1)
    oracle.set_threads(cores)
    return {
        "value": groups / step, "unit": UNIT, "cores": cores, "kind": "oracle",
        "sample": (f"fp64 C oracle, {cores} threads, bounded sample extrapolated to the step "
                   f"({W.tokens} tokens per input space, {groups} groups, window -{win[0]}/+{win[1]}): "
                   + "; ".join(samples) + f"; global scale + {init} codes over every whole matrix"),
        "single_thread_value": groups / step1,
        "single_thread_sample": "; ".join(samples1),
        "seconds_per_step": step,
        "hessian_tokens_channels_per_s": h_tc / max(step, 1e-30),
    }


def cpu_baseline_full(work: Work, win, single_thread_budget_s: float = 4.0) -> dict:
    """The fp64 oracle over the step's whole layer on all host cores, timed part by part
    (steady clock): the Hessian pass over every calibration chunk of every input space,
    then per matrix the global scale, the initial codes and the search with packing.  Each
    result is checked against the GPU's outputs of the step: h within 1e-4 relative; s_g
    bit for bit; codes and nibbles bit for bit in every group that is not an oracle near-tie
    (the search takes the GPU's fp32 h, so both sides search the same input).  X and W are
    copied to the host outside the timed parts.  One thread is timed on a bounded sample."""
    import oracle
    oracle.build()
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    oracle.set_threads(cores)
    down, up = win
    t_h = t_init = t_search = 0.0
    h_rel = 0.0
    tok_ch = 0
    for S in work.spaces.values():
        h_ref = np.zeros(S.n)
        for c in range(S.nchunks):
            xb = wl.bf16_bits(S.x[c * S.chunk:(c + 1) * S.chunk])
            t0 = time.perf_counter()
            oracle.hessian_accumulate(xb, h_ref)
            t_h += time.perf_counter() - t0
        tok_ch += S.tokens * S.n
        hg = S.h.double().cpu().numpy()
        h_rel = max(h_rel, float(np.max(np.abs(hg - h_ref) / np.maximum(h_ref, 1e-300))))
    mism = ties = groups = 0
    sg_ok = True
    for M in work.mats:
        wb = wl.bf16_bits(M.w)
        hg = M.space.h.cpu().numpy().astype(np.float32)
        t0 = time.perf_counter()
        s_g, _ = oracle.global_scale(wb)
        c0 = oracle.fourover6_codes(wb, s_g)[0] if work.init.startswith("4over6") else oracle.rtn_codes(wb, s_g)
        t_init += time.perf_counter() - t0
        t0 = time.perf_counter()
        ref = oracle.refine(wb, hg, s_g, c0, down, up)
        t_search += time.perf_counter() - t0
        sg_ok &= bool(np.float32(s_g) == np.float32(M.sg.item()))
        ok = ref["near_tie"] == 0
        codes = M.codes.cpu().numpy()
        packed = M.packed.cpu().numpy().reshape(M.m, M.n // 16, 8)
        bad = (codes != ref["codes"]) | np.any(packed != ref["packed"].reshape(M.m, M.n // 16, 8), axis=2)
        mism += int(np.count_nonzero(bad & ok))
        ties += int(np.count_nonzero(~ok))
        groups += M.groups
        del ref, wb
    total = t_h + t_init + t_search
    # one thread, bounded: the first chunk of the first input space and the first 64 rows of
    # every matrix, scaled to the whole layer by tokens and by rows
    oracle.set_threads(1)
    t1 = 0.0
    S0 = next(iter(work.spaces.values()))
    xb = wl.bf16_bits(S0.x[:S0.chunk])
    h1 = np.zeros(S0.n)
    t0 = time.perf_counter()
    oracle.hessian_accumulate(xb, h1)
    per_tc = (time.perf_counter() - t0) / (S0.chunk * S0.n)
    t1 += per_tc * tok_ch
    for M in work.mats:
        rows = min(M.m, 64)
        wb = wl.bf16_bits(M.w[:rows])
        s_g = np.float32(M.sg.item())
        t0 = time.perf_counter()
        c0 = oracle.rtn_codes(wb, s_g)
        oracle.refine(wb, M.space.h.cpu().numpy().astype(np.float32), s_g, c0, down, up)
        t1 += (time.perf_counter() - t0) * M.m / rows
    oracle.set_threads(cores)
    n_layers = work.W.n_layers
    return {
        "value": work.groups / total, "unit": UNIT, "cores": cores, "kind": "oracle",
        "sample": (f"full: the fp64 C oracle over the whole layer ({work.W.name} layer 0: {work.groups} groups, "
                   f"{tok_ch} token-channels of X, window -{down}/+{up}, {work.init} start) on {cores} threads, "
                   f"steady-clock timed: Hessian pass {t_h:.2f} s, global scale + initial codes {t_init:.2f} s, "
                   f"search + pack {t_search:.2f} s"
                   + (f"; per model {n_layers} layers, extrapolated x{n_layers}: {total * n_layers:.1f} s"
                      if n_layers > 1 else "")),
        "seconds_per_layer": total,
        "seconds_per_model": total * n_layers if n_layers > 1 else None,
        "seconds_per_model_note": f"extrapolated x{n_layers} from layer 0" if n_layers > 1 else None,
        "phases_s": {"hessian": t_h, "init": t_init, "search": t_search},
        "hessian_tokens_channels_per_s": tok_ch / t_h if t_h > 0 else None,
        "search_groups_per_s": groups / t_search if t_search > 0 else None,
        "verified": {"h_max_rel_err": h_rel, "h_ok": h_rel <= 1e-4, "global_scale_bit_exact": sg_ok,
                     "groups": groups, "near_ties": ties, "mismatches_outside_near_ties": mism},
        "single_thread_value": work.groups / t1,
        "single_thread_sample": ("one thread on a bounded sample extrapolated to the layer: the first "
                                 f"{S0.chunk}-token chunk of {S0.name} (scaled by token-channels) and the "
                                 "first 64 rows of every matrix (scaled by rows)"),
    }


def reference_arm(args, d: Dist):
    """--impl reference: the CPU oracle, as it stands, on the host cores."""
    if d.rank != 0:
        return
    import oracle
    oracle.build()
    W = wl.WORKLOADS[args.workload]
    win = window_of(args, W)
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    vals = []
    samples = []
    for i in range(args.warmup + args.steps):
        step, _, samples, _ = _oracle_step(W, win, 3.0, args.init, cores)
        if i >= args.warmup:
            vals.append(step)
    groups = sum(L.out_features * L.in_features // 16 for L in W.layers)
    sec = statistics.mean(vals)
    value = groups / sec
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": sec * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": W.name, "matrices": [[L.name, L.out_features, L.in_features] for L in W.layers],
                   "tokens": W.tokens, "window": list(win), "init": args.init},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": (f"fp64 C oracle, {cores} threads, per step a bounded sample extrapolated "
                                    f"to the step ({W.tokens} tokens per input space, {groups} groups, window "
                                    f"-{win[0]}/+{win[1]}): " + "; ".join(samples)
                                    + f"; global scale + {args.init} codes over every whole matrix")},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def output_error_eval(hs, work: Work, peaks: dict, tokens: int = 8192, reps: int = 5):
    """Layer-output error ||X dW^T||_F^2 (Eq. 3) of the first matrix on one chunk of its
    calibration tokens, for the RTN codes and for the searched codes of the step, on the
    tensor cores; with the GEMM's throughput.  Outside the timed step."""
    M = work.mats[0]
    S = M.space
    T = min(tokens, S.tokens)
    x = S.x[:T]
    dev = x.device
    ld = hs.residual_ld(M.n)
    dw2 = torch.empty(M.m, ld, dtype=torch.bfloat16, device=dev)
    out = torch.zeros(1, dtype=torch.float64, device=dev)
    ws = torch.empty(hs.hscale_output_error_workspace_bytes(T, M.m), dtype=torch.uint8, device=dev)
    rtn_codes = torch.empty_like(M.codes)
    rtn_packed = torch.empty_like(M.packed)
    hs.hscale_rtn_scales(M.w, M.sg, rtn_codes, work.ws)
    hs.hscale_pack_nvfp4(M.w, M.sg, rtn_codes, rtn_packed)
    err = {}
    for name, codes, packed in (("rtn", rtn_codes, rtn_packed), ("hscale", M.codes, M.packed)):
        hs.hscale_dequant_residual(M.w, M.sg, codes, packed, dw2)
        out.zero_()
        hs.hscale_output_error(x, dw2, M.m, out, ws)
        err[name] = float(out.item())
    ms = timed(lambda: hs.hscale_output_error(x, dw2, M.m, out, ws), reps)
    ms_res = timed(lambda: hs.hscale_dequant_residual(M.w, M.sg, M.codes, M.packed, dw2), reps)
    n_pad = ld // 2
    executed = 2.0 * T * M.m * (2 * n_pad)        # X [hi | lo]^T: K = 2 n_pad
    useful = 2.0 * T * M.m * M.n                  # X dW^T
    peak = float(peaks.get("bf16_tflops", 1900.0))
    return {"matrix": M.name, "tokens": T, "error_rtn": err["rtn"], "error_hscale": err["hscale"],
            "reduction": 1.0 - err["hscale"] / err["rtn"] if err["rtn"] > 0 else None,
            "gemm_ms": ms, "gemm_tflops_executed": executed / (ms * 1e-3) / 1e12,
            "gemm_tflops_useful": useful / (ms * 1e-3) / 1e12,
            "frac_of_measured_bf16": executed / (ms * 1e-3) / 1e12 / peak, "bf16_peak_tflops": peak,
            "residual_ms": ms_res,
            "note": "tcgen05 bf16 GEMM of X with the [hi | lo] split of dW, fused sum of squares"}


def gptq_eval(hs, work: Work, peaks: dict, block: int = 128, reps: int = 3):
    """Algorithm 3 (GPTQ + H-Scale) on the first matrix of the workload, outside the timed
    step: the full Hessian X^T X over every calibration chunk of its input space on the
    tensor cores, the damped inverse-Cholesky factor, and the block loop with H-Scale as the
    local quantizer (blocks of `block` columns, the step's window); each timed, and the
    layer-output error ||X dW^T||^2 on the first chunk for GPTQ + H-Scale, H-Scale and RTN."""
    M = work.mats[0]
    S = M.space
    dev = S.x.device
    n, m = M.n, M.m
    down, up = work.win
    H = torch.zeros(n, n, dtype=torch.float32, device=dev)
    # one call over every token: the kernel accumulates 2048-token segments whatever the
    # call, so a large call costs no accuracy and saves per-launch work; X's rows are
    # 16-byte aligned, so it is read as it is (no workspace)
    call = S.tokens

    def hessian():
        H.zero_()
        for t0 in range(0, S.tokens, call):
            hs.hscale_hessian_full_accumulate(S.x[t0:t0 + call], H)

    ms_h = timed(hessian, reps)
    U = torch.empty(n, n, dtype=torch.float32, device=dev)
    dead = torch.empty(n, dtype=torch.uint8, device=dev)
    info = torch.zeros(3, dtype=torch.int32, device=dev)
    fws = torch.empty(max(256, hs.hscale_gptq_factor_workspace_bytes(n)), dtype=torch.uint8, device=dev)
    ms_f = timed_graph(lambda: hs.hscale_gptq_factor(H, 0.01, U, dead, info, fws), reps)
    if int(info.abs().sum().item()) != 0:
        return {"unavailable": f"factorization failed, info {info.tolist()}"}
    h = torch.diagonal(H).contiguous()
    codes = torch.empty_like(M.codes)
    packed = torch.empty_like(M.packed)
    gws = torch.empty(hs.hscale_gptq_workspace_bytes(m, n, block), dtype=torch.uint8, device=dev)
    ms_q = timed_graph(lambda: hs.hscale_gptq_hscale(M.w, U, h, M.sg, dead, block, down, up, codes, packed, gws),
                       reps)
    # output error on the first chunk: GPTQ + H-Scale, H-Scale (the step's outputs), RTN
    T = S.chunk
    x = S.x[:T]
    dw2 = torch.empty(m, hs.residual_ld(n), dtype=torch.bfloat16, device=dev)
    out = torch.zeros(1, dtype=torch.float64, device=dev)
    ows = torch.empty(hs.hscale_output_error_workspace_bytes(T, m), dtype=torch.uint8, device=dev)
    rtn_codes = torch.empty_like(M.codes)
    rtn_packed = torch.empty_like(M.packed)
    hs.hscale_rtn_scales(M.w, M.sg, rtn_codes, work.ws)
    hs.hscale_pack_nvfp4(M.w, M.sg, rtn_codes, rtn_packed)
    err = {}
    for name, c, p in (("gptq_hscale", codes, packed), ("hscale", M.codes, M.packed), ("rtn", rtn_codes, rtn_packed)):
        hs.hscale_dequant_residual(M.w, M.sg, c, p, dw2)
        out.zero_()
        hs.hscale_output_error(x, dw2, m, out, ows)
        err[name] = float(out.item())
    h_flop = 2.0 * S.tokens * n * n
    # the 128 x 256 output tiles the GEMM computes (those wholly below the diagonal are skipped)
    tiles = sum(1 for tm in range((n + 127) // 128) for tn in range((n + 255) // 256) if (tn + 1) * 256 > tm * 128)
    h_flop_done = 2.0 * S.tokens * 128 * 256 * tiles
    upd_flop = sum(2.0 * m * block * (n - c0 - block) for c0 in range(0, n, block))
    peak = float(peaks.get("bf16_tflops", 1900.0))
    return {"matrix": M.name, "block": block, "window": [down, up], "tokens": S.tokens,
            "timing": "the full Hessian as eager calls; the factor and the block loop (about 200 and 300 "
                      "dependent launches per call) captured once as CUDA graphs and replayed",
            "hessian_full_ms": ms_h, "hessian_full_tflops": h_flop / (ms_h * 1e-3) / 1e12,
            "hessian_full_note": "dense-equivalent 2 T n^2 FLOP; tiles wholly below the diagonal are skipped, "
                                 "so the computed-tile rate below is the one to compare with the peak; X is read "
                                 "as it is (MN-major operand tiles, no transpose)",
            "hessian_full_tokens_per_call": call,
            "hessian_full_tflops_computed": h_flop_done / (ms_h * 1e-3) / 1e12,
            "hessian_full_frac_of_measured_bf16": h_flop_done / (ms_h * 1e-3) / 1e12 / peak,
            "factor_ms": ms_f, "block_loop_ms": ms_q, "update_gemm_gflop": upd_flop / 1e9,
            "output_error_chunk_tokens": T, "output_error": err,
            "reduction_vs_rtn": 1.0 - err["gptq_hscale"] / err["rtn"],
            "reduction_vs_hscale": 1.0 - err["gptq_hscale"] / err["hscale"]}


def shift_statistics(work: Work, win, sample_rows: int = 16):
    """Selected shifts delta = chosen code - initial code over every group of the step
    (from the GPU outputs), and the mean reduction of the Hessian-weighted error per
    delta relative to delta = 0 on a sample of rows (from the CPU oracle).  The paper
    reports the same statistics for real weights (Sec. 4, selected scale shifts)."""
    down, up = win
    hist = torch.zeros(down + up + 1, dtype=torch.int64)
    for M in work.mats:
        delta = M.codes.to(torch.int16) - M.codes0.to(torch.int16)
        hist += torch.bincount((delta.flatten() + down).clamp(0, down + up).to(torch.int64).cpu(),
                               minlength=down + up + 1)
    total = int(hist.sum())
    out = {"window": [down, up], "groups": total,
           "delta_hist": {str(i - down): int(v) for i, v in enumerate(hist.tolist())},
           "keep": float(hist[down]) / total, "larger": float(hist[down + 1:].sum()) / total,
           "smaller": float(hist[:down].sum()) / total}
    try:
        import oracle
        M = work.mats[0]
        rows = np.linspace(0, M.m - 1, num=min(sample_rows, M.m)).astype(int)
        ref = oracle.refine(wl.bf16_bits(M.w[rows]), M.space.h.cpu().numpy(), M.sg.item(),
                            M.codes0[rows].cpu().numpy(), down, up)
        red = {}
        for dlt in range(-down, up + 1):
            sel = ref["delta"] == dlt
            if sel.any() and dlt != 0:
                e0, e1 = ref["e_init"][sel], ref["e_best"][sel]
                ok = e0 > 0
                red[str(dlt)] = float(np.mean(1.0 - e1[ok] / e0[ok])) if ok.any() else None
        tot0, tot1 = ref["e_init"].sum(), ref["e_best"].sum()
        out["mean_error_reduction_by_delta"] = red
        out["error_removed"] = float(1.0 - tot1 / tot0) if tot0 > 0 else None
        out["error_sample"] = f"oracle on {rows.size} rows of {M.name}"
    except Exception as e:  # the statistics are context; never fail the run for them
        out["error_sample"] = f"unavailable: {e}"
    return out


# ------------------------------------------------------------------ GPU arm
def measure_workload(hs, d: Dist, args, W: wl.Workload, win, dev, overlap_ctas: int, pipeline: str,
                     tokens=None, init="rtn", col_block=0):
    """One workload's timed steps (CUDA graphs, max over ranks), the Hessian and search
    figures, and the search over every window of the workload timed per kernel.  Returns
    (result dict, work); the work keeps the step's outputs."""
    work = Work(W, d.rank, win, dev, tokens=tokens, init=init, col_block=col_block)
    work.search_schedule = args.search_schedule
    work.weight_pass = args.weight_pass
    work.ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev)
    torch.cuda.synchronize()

    warm = max(args.warmup, 3)
    for _ in range(warm):
        run_step(hs, work)
    torch.cuda.synchronize()

    # eager launches (one API call per chunk and matrix), for reference
    ms_eager = timed(lambda: run_step(hs, work), args.steps)

    # timed region: the same launches replayed from CUDA graphs
    pipelined = work.pipelined(pipeline)
    overlap = work.overlap_ctas(overlap_ctas, pipelined)
    graphs = StepGraphs(hs, work, overlap, pipeline=pipelined)
    for _ in range(warm):
        graphs.replay()
    graphs.drain()
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    d.barrier()
    torch.cuda.synchronize()
    with ClockSampler(d.local) as clk:
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record()
        for s in range(args.steps):
            graphs.replay(evs[s])
        graphs.drain()
        t1.record()
        torch.cuda.synchronize()
    d.barrier()
    ms_total = t0.elapsed_time(t1)
    ms_h = sum(e[0].elapsed_time(e[1]) for e in evs) / args.steps
    ms_sc = sum(e[1].elapsed_time(e[2]) for e in evs) / args.steps
    ms_step = d.max(ms_total / args.steps)

    # ---- per-kernel times of the scale phase, every matrix, every window of the workload
    hbm_peak, peak_kind, peaks = measured_peaks()
    props = torch.cuda.get_device_properties(dev)
    sm_max_mhz = float(peaks.get("sm_max_mhz", 2070.0))
    fp32_peak = props.multi_processor_count * 128 * sm_max_mhz * 1e6
    reps = max(3, min(args.steps, 20))
    # W of a matrix can be smaller than L2: its kernels are timed after an L2 flush (twice
    # the L2 size written, then another twice read, between calls, outside the timed window)
    l2 = int(getattr(props, "L2_cache_size", 0) or (126 << 20))
    flush = (torch.empty(2 * l2 // 4, dtype=torch.float32, device=dev),
             torch.zeros(2 * l2 // 4, dtype=torch.float32, device=dev))
    ms_init = sum(timed(lambda M=M: init_codes(hs, work, M), reps, flush) for M in work.mats)
    ms_h_alone = timed(lambda: [g.replay() for g in graphs.gh[0]], reps)
    sweep = []
    windows = sorted(set([tuple(win)] + [(kk, kk) for kk in W.window]))
    for dn, upw in windows:
        ms_ref = 0.0
        for M in work.mats:
            ms_ref += timed(lambda M=M: refine(hs, work, M, dn, upw), reps, flush)
        C = dn + upw + 1
        t_bytes = SEARCH_BYTES[work.init] * work.groups / (hbm_peak * 1e9)
        t_ops = 80 * C * work.groups / fp32_peak
        sweep.append({"window": [dn, upw], "candidates": C, "ms": ms_ref,
                      "groups_per_s": work.groups / (ms_ref * 1e-3),
                      "bound": "alu" if t_ops > t_bytes else "hbm", "roofline_ms": max(t_bytes, t_ops) * 1e3,
                      "frac": max(t_bytes, t_ops) / (ms_ref * 1e-3)})
    del flush
    # restore the outputs of the step's own window; materialize the initial codes the
    # search decided inline, for the shift statistics
    scale_phase(hs, work)
    for M in work.mats:
        if work.init == "rtn":
            hs.hscale_rtn_scales(M.w, M.sg, M.codes0, work.ws)
        elif work.init == "4over6":
            hs.hscale_fourover6_codes(M.w, M.sg, M.codes0)
    torch.cuda.synchronize()
    main = [s for s in sweep if tuple(s["window"]) == tuple(win)][0]

    # ---- roofline of the Hessian pass: algorithmic bytes over the launches' event time
    h_bytes_launch = work.h_bytes / work.h_launches
    ms_h_launch = ms_h / work.h_launches
    h_gbs = work.h_bytes / (ms_h * 1e-3) / 1e9
    traffic = step_traffic(work)
    hess_roof = {"bound": "hbm", "kernel": "hessian_colsumsq", "achieved": h_gbs,
                 "peak": hbm_peak, "unit": "GB/s", "frac": h_gbs / hbm_peak,
                 "peak_kind": f"{peak_kind} HBM copy bandwidth",
                 "frac_of_8TBs_spec": h_gbs / HBM_SPEC_GBS, "traffic": traffic,
                 "bytes_per_launch": h_bytes_launch, "ms_per_launch": ms_h_launch}
    # ---- roofline of the search (its own window, W read from HBM after an L2 flush)
    if main["bound"] == "alu":
        ops = 80.0 * main["candidates"] * work.groups
        search_roof = {"bound": "alu", "kernel": SEARCH_KERNELS, "achieved": ops / (main["ms"] * 1e-3) / 1e12,
                       "peak": fp32_peak / 1e12, "unit": "Tops/s", "frac": main["frac"],
                       "peak_kind": "SMs x 128 fp32 lanes x max SM clock; 5 lane operations per element "
                                    "and candidate", "candidates": main["candidates"], "traffic": None,
                       "ops_per_launch": ops / len(work.mats), "ms_per_launch": main["ms"] / len(work.mats)}
    else:
        b = SEARCH_BYTES[work.init] * work.groups
        search_roof = {"bound": "hbm", "kernel": SEARCH_KERNELS, "achieved": b / (main["ms"] * 1e-3) / 1e9,
                       "peak": hbm_peak, "unit": "GB/s", "frac": b / (main["ms"] * 1e-3) / 1e9 / hbm_peak,
                       "peak_kind": f"{peak_kind} HBM copy bandwidth", "candidates": main["candidates"],
                       "traffic": None, "bytes_per_launch": b / len(work.mats),
                       "ms_per_launch": main["ms"] / len(work.mats)}
    # the dominant kernel of the step: the Hessian pass, unless the searches take longer
    # than the Hessian passes do alone (e.g. the 70B MLP block)
    dominant = search_roof if main["ms"] > ms_h_alone else hess_roof
    res = {
        "work": work, "graphs": graphs, "ms_step": ms_step, "ms_eager": ms_eager, "warm": warm,
        "value": work.groups * d.world / (ms_step * 1e-3), "overlap_ctas": overlap,
        "search_schedule": work.search_schedule,
        "roofline": dominant, "roofline_hessian": hess_roof, "roofline_search": search_roof,
        "step_hbm": step_hbm(work, ms_step, hbm_peak, peak_kind),
        "phases_ms": {"hessian": ms_h, "after_hessian": ms_sc, "hessian_alone": ms_h_alone,
                      "weight_only": ms_init, "refine": main["ms"]},
        "hessian": {"gbs": h_gbs, "tokens_channels_per_s": work.h_bytes / 2 / (ms_h * 1e-3),
                    "frac_of_measured_hbm": h_gbs / hbm_peak, "frac_of_8TBs": h_gbs / HBM_SPEC_GBS},
        "search": {"groups_per_s": main["groups_per_s"], "candidates": main["candidates"],
                   "bound": main["bound"], "roofline_s": main["roofline_ms"] * 1e-3, "frac": main["frac"],
                   "fp32_peak_ops": fp32_peak, "sm_count": props.multi_processor_count,
                   "clock_mhz_for_peak": sm_max_mhz},
        "sweep": sweep, "clocks": clk.summary(), "peaks": peaks,
    }
    return res, work


def compact_roofline(r: dict) -> dict:
    """The figures of a roofline object that a one-line summary needs."""
    return {k: r[k] for k in ("kernel", "bound", "achieved", "peak", "unit", "frac") if k in r}


def extra_workload(hs, d: Dist, args, name: str, dev) -> dict:
    """A second workload measured in the same process (its own timed steps and its search
    over every window of the workload): per-step time, the step's rate and both rooflines,
    and the window sweep."""
    W = wl.WORKLOADS[name]
    res, work = measure_workload(hs, d, args, W, (W.window[0], W.window[0]), dev, -1, "auto")
    out = {"workload": W.name, "matrices": [[M.name, M.m, M.n] for M in work.mats],
           "input_spaces": [[S.name, S.tokens, S.n, S.chunk] for S in work.spaces.values()],
           "window": [W.window[0], W.window[0]], "groups": work.groups,
           "ms_per_step": res["ms_step"], "value": res["value"], "unit": UNIT,
           "schedule": "pipelined" if res["graphs"].pipeline else "sequential",
           "weight_pass": res["work"].weight_pass,
           "roofline_hessian": compact_roofline(res["roofline_hessian"]),
           "roofline_search": compact_roofline(res["roofline_search"]),
           "step_hbm": {k: res["step_hbm"][k] for k in ("bytes", "achieved", "peak", "unit", "frac")},
           "phases_ms": res["phases_ms"], "clocks": res["clocks"],
           "search_sweep": [{k: s[k] for k in ("window", "candidates", "ms", "groups_per_s", "bound", "frac")}
                            for s in res["sweep"]]}
    del res, work
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    return out


def gpu_arm(args, d: Dist):
    import paper_2608_28113_gb300 as hs
    hs.load()
    torch.cuda.set_device(d.local)
    dev = torch.device("cuda", d.local)
    W = wl.WORKLOADS[args.workload]
    win = window_of(args, W)
    res, work = measure_workload(hs, d, args, W, win, dev, args.overlap_ctas, args.pipeline,
                                 tokens=args.tokens, init=args.init, col_block=args.col_block)
    graphs, peaks, ms_step = res["graphs"], res["peaks"], res["ms_step"]
    shifts = shift_statistics(work, win)
    out_err = None if args.no_output_error else output_error_eval(hs, work, peaks)
    gptq = None
    if not args.no_gptq:
        try:
            gptq = gptq_eval(hs, work, peaks)
        except Exception as e:  # report, keep the bench line
            gptq = {"unavailable": f"{type(e).__name__}: {e}"}

    # ---- end to end through the public API with host buffers
    e2e = None if args.no_e2e else e2e_leg(hs, work, args)

    n_layers = W.n_layers
    roofline = dict(res["roofline"])
    # the other kernel's roofline in the same object, so a reader of the standard keys sees
    # both targets of the path
    other = res["roofline_search"] if roofline["kernel"] == "hessian_colsumsq" else res["roofline_hessian"]
    roofline["other"] = compact_roofline(other)
    line = {
        "metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": d.world, "steps": args.steps,
        "warmup": res["warm"], "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "input_dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": W.name,
                   "matrices": [[M.name, M.m, M.n] for M in work.mats],
                   "input_spaces": [[S.name, S.tokens, S.n, S.chunk] for S in work.spaces.values()],
                   "window": list(win), "init": work.init, "groups": work.groups,
                   "col_block": work.col_block,
                   "schedule": "pipelined" if graphs.pipeline else "sequential",
                   "weight_pass": work.weight_pass,
                   "l2": "inputs larger than L2: %.2f GB of X streamed per step" %
                         (sum(S.tokens * S.n * 2 for S in work.spaces.values()) / 1e9),
                   "parallelism": f"independent layer per GPU x{d.world}"},
        "roofline": roofline,
        "roofline_search": res["roofline_search"],
        "roofline_hessian": res["roofline_hessian"],
        "step_hbm": res["step_hbm"],
        "seconds_per_layer": ms_step * 1e-3,
    }
    if n_layers > 1:
        line["seconds_per_model"] = ms_step * 1e-3 * n_layers
        line["seconds_per_model_note"] = f"{n_layers} layers of identical shapes: per-layer step x {n_layers}"
    line.update({
        "phases_ms": res["phases_ms"],
        "ms_per_step_eager": res["ms_eager"],
        "timed_launch": ("CUDA graphs of the step's API calls on three streams: the Hessian pass of "
                         + (f"each {work.col_block}-channel column block of each input space over every token"
                            if work.col_block else "each input space in token chunks")
                         + "; alongside it the weight-only calls (s_g, 4over6 codes); the searches of "
                         + ("each block" if work.col_block else "each input space")
                         + " as soon as its h is complete"
                         + (f" (at most {res['overlap_ctas']} search CTAs per SM while a Hessian pass runs)"
                            if res["overlap_ctas"] > 0 and (len(work.pieces) > 1 or graphs.pipeline) else "")
                         + ("; consecutive steps pipelined: each step's last searches run alongside the next "
                            "step's first Hessian pass (h, s_g and initial codes double-buffered); the timed "
                            "region ends when the last step's searches are done" if graphs.pipeline else "")),
        "hessian": res["hessian"],
        "search": res["search"],
        "clocks": res["clocks"],
        "gpu_launches": args.steps * (work.h_launches + kernels_per_matrix(work) * len(work.mats)),
    })
    if len(res["sweep"]) > 1:
        line["search_sweep"] = res["sweep"]
    line["shift_statistics"] = shifts
    if out_err:
        line["output_error"] = out_err
    if gptq:
        line["gptq_hscale"] = gptq
    if e2e:
        line["e2e"] = e2e
    if d.rank == 0 and d.world == 1 and not args.no_cpu_baseline:
        if args.cpu_baseline == "full" and work.col_block == 0:
            line["cpu_baseline"] = cpu_baseline_full(work, win)
        else:
            cb = cpu_baseline(W, win, init=args.init)
            line["cpu_baseline"] = {k2: cb[k2] for k2 in ("value", "unit", "cores", "kind", "sample",
                                                          "single_thread_value")}
    # a second workload from the same process (the 70B MLP block with its window sweep)
    if args.extra_workload != "none" and args.extra_workload != W.name:
        del graphs, res, work
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        line[args.extra_workload.replace("-", "_")] = extra_workload(hs, d, args, args.extra_workload, dev)
    if d.rank == 0:
        print(json.dumps(line), flush=True)


def e2e_leg(hs, work: Work, args):
    """Whole step through the public API with host buffers: X chunks and W copied from
    pinned host memory inside the timed region (chunk copies on a copy stream overlap
    the Hessian pass), codes and nibbles copied back."""
    dev = next(iter(work.spaces.values())).x.device
    x_host, xbuf = {}, {}
    nbuf = 3
    for S in work.spaces.values():
        x_host[S.name] = torch.empty(S.x.shape, dtype=S.x.dtype, pin_memory=True)
        x_host[S.name].copy_(S.x)
        xbuf[S.name] = [torch.empty(S.chunk, S.n, dtype=torch.bfloat16, device=dev) for _ in range(nbuf)]
    w_host = {M.name: torch.empty(M.w.shape, dtype=M.w.dtype, pin_memory=True).copy_(M.w) for M in work.mats}
    w_dev = {M.name: torch.empty_like(M.w) for M in work.mats}
    out_host = {M.name: (torch.empty(M.codes.shape, dtype=torch.uint8, pin_memory=True),
                         torch.empty(M.packed.shape, dtype=torch.uint8, pin_memory=True)) for M in work.mats}
    copy = torch.cuda.Stream(device=dev)
    comp = torch.cuda.current_stream(dev)

    def step():
        # the copies of this step start after the previous step's kernels are done with the
        # staging buffers
        copy.wait_stream(comp)
        for S in work.spaces.values():
            done = [torch.cuda.Event() for _ in range(nbuf)]
            S.h.zero_()
            for c in range(S.nchunks):
                b = c % nbuf
                with torch.cuda.stream(copy):
                    if c >= nbuf:
                        copy.wait_event(done[b])
                    xbuf[S.name][b].copy_(x_host[S.name][c * S.chunk:(c + 1) * S.chunk], non_blocking=True)
                    ready = torch.cuda.Event()
                    ready.record(copy)
                comp.wait_event(ready)
                hs.hscale_hessian_diag_accumulate(xbuf[S.name][b], S.h)
                done[b].record(comp)
        with torch.cuda.stream(copy):
            for M in work.mats:
                w_dev[M.name].copy_(w_host[M.name], non_blocking=True)
            wr = torch.cuda.Event()
            wr.record(copy)
        comp.wait_event(wr)
        scale_phase(hs, work, ws=w_dev)
        for M in work.mats:
            out_host[M.name][0].copy_(M.codes, non_blocking=True)
            out_host[M.name][1].copy_(M.packed, non_blocking=True)

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    # per-step times: the host link is shared with the machine's other jobs, and a busy
    # moment can stretch single steps 2-4x, so the median step is reported (mean and best
    # beside it)
    reps = max(5, min(args.steps, 10))
    step_ms = []
    for _ in range(reps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        step()
        e1.record()
        torch.cuda.synchronize()
        step_ms.append(e0.elapsed_time(e1))
    ms = statistics.median(step_ms)
    h2d = sum(S.tokens * S.n * 2 for S in work.spaces.values()) + sum(M.m * M.n * 2 for M in work.mats)
    d2h = sum(M.codes.numel() + M.packed.numel() for M in work.mats)
    # the host link on these very buffers: the step's host -> device bytes as plain copies
    # (X into its resident copy, the same values; W into its staging buffer), best of 3
    def copies_only():
        for S in work.spaces.values():
            S.x.copy_(x_host[S.name], non_blocking=True)
        for M in work.mats:
            w_dev[M.name].copy_(w_host[M.name], non_blocking=True)

    best = float("inf")
    for _ in range(3):
        best = min(best, timed(copies_only, 1))
    return {"value": work.groups / (ms * 1e-3), "unit": UNIT, "ms_per_step": ms,
            "ms_per_step_mean": statistics.mean(step_ms), "ms_per_step_best": min(step_ms), "steps_timed": reps,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "copies_only_ms": best, "h2d_link_gbs": h2d / (best * 1e-3) / 1e9, "frac_of_link_bound": best / ms}


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
