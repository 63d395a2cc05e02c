"""The bench's step schedule.  On the CPU: the flow-shop order of the input spaces, the
column blocks and Hessian calls of a piece, and the pipelining and overlap policies.  On
the GPU: the graph schedule reproduces an eager pass."""
import itertools
import os
import random
import sys
from types import SimpleNamespace

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def makespan(order, jobs):
    """Two-machine flow shop: stage 1 of each job in turn on machine 1, stage 2 on
    machine 2 once its stage 1 is done and machine 2 is free."""
    t1 = t2 = 0.0
    for name in order:
        _, a, b = jobs[name]
        t1 += a
        t2 = max(t2, t1) + b
    return t2


def test_johnson_order_minimises_the_makespan():
    rng = random.Random(5)
    for _ in range(200):
        n = rng.randint(1, 6)
        jobs = {f"j{i}": (f"j{i}", rng.uniform(0.1, 3.0), rng.uniform(0.1, 3.0)) for i in range(n)}
        order = bench.johnson_order(list(jobs.values()))
        assert sorted(order) == sorted(jobs)
        best = min(makespan(p, jobs) for p in itertools.permutations(jobs))
        assert makespan(order, jobs) <= best + 1e-12


def test_column_blocks_and_hessian_calls_cover_the_space_once():
    S = SimpleNamespace(n=4096, chunk=8192, tokens=8192 * 32)
    assert bench.column_blocks(S, 0) == [(0, 4096)]
    assert bench.column_blocks(S, 4096) == [(0, 4096)]
    blocks = bench.column_blocks(S, 1536)
    assert blocks == [(0, 1536), (1536, 3072), (3072, 4096)]
    for c0, c1 in blocks + [(0, 4096)]:
        calls = bench.hessian_calls(S, c0, c1)
        assert calls[0][0] == 0 and calls[-1][1] == S.tokens
        assert all(a[1] == b[0] for a, b in zip(calls, calls[1:]))
        # a launch reads about a chunk's bytes: more rows when the block is narrower
        assert all(t1 - t0 <= max(S.chunk, S.chunk * S.n // (c1 - c0)) for t0, t1 in calls)


def fake_work(spaces, mats, win=(4, 4)):
    """A Work with only what the schedule policies read: spaces (name -> tokens, n) and
    matrices (groups, space name)."""
    w = bench.Work.__new__(bench.Work)
    w.win = win
    w.spaces = {name: SimpleNamespace(name=name, tokens=t, n=n) for name, (t, n) in spaces.items()}
    w.mats = [SimpleNamespace(groups=g, space=w.spaces[s]) for g, s in mats]
    return w


def test_pipelining_and_overlap_policies():
    # one Hessian-bound input space (q_proj): pipelined unless asked not to, 4 search CTAs
    q = fake_work({"x": (262144, 4096)}, [(4096 * 4096 // 16, "x")])
    assert not q.search_bound()
    assert q.pipelined("auto") and q.pipelined("on") and not q.pipelined("off")
    assert q.overlap_ctas(-1, True) == 4 and q.overlap_ctas(-1, False) == 4 and q.overlap_ctas(2, False) == 2
    # several input spaces (decoder layer): pipelined
    dec = fake_work({"qkv": (131072, 4096), "o": (131072, 4096), "mlp": (131072, 4096),
                     "down": (131072, 14336)},
                    [(1 << 20, "qkv"), (1 << 18, "qkv"), (1 << 18, "qkv"), (1 << 20, "o"),
                     (3670016, "mlp"), (3670016, "mlp"), (3670016, "down")])
    assert not dec.search_bound() and dec.pipelined("auto") and dec.overlap_ctas(-1, True) == 4
    assert not dec.pipelined("off")
    # one input space but search-bound (a wide window over a large matrix): pipelined, the
    # searches fill the SMs
    wide = fake_work({"x": (65536, 8192)}, [(28672 * 8192 // 16, "x")] * 2, win=(16, 16))
    assert wide.search_bound() and wide.pipelined("auto")
    assert wide.overlap_ctas(-1, True) == 7 and wide.overlap_ctas(-1, False) == 7


@pytest.mark.gpu
@pytest.mark.parametrize("workload,pipeline", [("llama8b-decoder", True), ("llama8b-decoder", False),
                                               ("llama8b-q_proj", True)])
def test_step_graphs_reproduce_the_eager_step(workload, pipeline):
    """The bench's graph schedule (three streams; with pipelining, consecutive steps
    overlapping on two buffer sets) gives the outputs of one eager pass, in every buffer
    set, after several steps."""
    import torch

    import paper_2608_28113_gb300 as hs
    from paper_2608_28113_gb300 import workloads as wl

    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()
    dev = torch.device("cuda", 0)
    W = wl.WORKLOADS[workload]
    work = bench.Work(W, 0, (4, 4), dev, tokens=16384)
    work.ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev)
    bench.run_step(hs, work)
    torch.cuda.synchronize()
    ref = [(M.codes.clone(), M.packed.clone(), M.sg.clone()) for M in work.mats]
    ref_h = {S.name: S.h.clone() for S in work.spaces.values()}
    graphs = bench.StepGraphs(hs, work, 4, pipeline=pipeline)
    assert graphs.pipeline == pipeline and len(graphs.sets) == (2 if pipeline else 1)
    for i in range(len(graphs.sets)):
        graphs.bind(i)
        for S in work.spaces.values():
            S.h.fill_(-1.0)
        for M in work.mats:
            M.sg.fill_(-1.0)
    graphs.bind(0)
    for M in work.mats:
        M.codes.zero_()
        M.packed.zero_()
    for _ in range(5):
        graphs.replay()
    graphs.drain()
    torch.cuda.synchronize()
    for M, (c, p, sg) in zip(work.mats, ref, strict=True):
        assert torch.equal(M.codes, c) and torch.equal(M.packed, p)
    for i in range(len(graphs.sets)):
        graphs.bind(i)
        for S in work.spaces.values():
            assert torch.equal(S.h, ref_h[S.name])
        for M, (_, _, sg) in zip(work.mats, ref, strict=True):
            assert torch.equal(M.sg, sg)
    graphs.bind(0)


def test_search_schedule_policy():
    """--search-schedule: 'auto' passes the work-sharing workspace to every search except
    one that fills the SMs (7 CTAs each) beside a Hessian pass; 'shared' and 'static'
    always and never."""
    w = SimpleNamespace(search_schedule="auto")
    assert bench.shares(w, 0) and bench.shares(w, 4) and bench.shares(w, 6)
    assert not bench.shares(w, 7) and not bench.shares(w, 8)
    w.search_schedule = "shared"
    assert all(bench.shares(w, c) for c in (0, 4, 7))
    w.search_schedule = "static"
    assert not any(bench.shares(w, c) for c in (0, 4, 7))


def test_step_hbm_counts_every_byte_of_the_step():
    """The whole-step HBM figure: X's bytes of the Hessian passes, W once for the global
    amax and once in the search (again for the two-pass 4over6 codes), and the codes and
    nibbles written; per group 32 + 41, or 65 + 42 with the two-pass init."""
    work = SimpleNamespace(h_bytes=6_000_000, groups=1000, init="rtn")
    r = bench.step_hbm(work, ms_step=1.0, hbm_peak=6000.0, peak_kind="measured")
    assert r["bytes"] == 6_000_000 + 73 * 1000
    assert abs(r["achieved"] - r["bytes"] / 1e-3 / 1e9) < 1e-9
    assert abs(r["frac"] - r["achieved"] / 6000.0) < 1e-12
    work.init = "4over6-2pass"
    assert bench.step_hbm(work, 1.0, 6000.0, "measured")["bytes"] == 6_000_000 + 107 * 1000
