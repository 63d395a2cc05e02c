"""The CUDA side of the sharded path (paper_2608_28113_gb300.sharded): the entry points a
token- or row-sharded run needs, with the ranks emulated in one process on one GPU.

* hscale_hessian_sum_partials: the rank-order sum of per-share partial h equals the one-pass
  h within 1e-4 and the oracle's fp64 h within 1e-4; it is the same bits on every call.
* hscale_amax_bits + hscale_global_scale_from_amax: the maximum of the row shares' words gives
  the s_g of hscale_rtn_scales over the whole matrix, bit for bit (also all-zero and
  exact-tie matrices, and an empty shard).
* the search of each row share with that s_g gives the whole-matrix search's bytes.
* quantize_layer_sharded without a process group is the one-rank path.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2608_28113_gb300 as hs
from paper_2608_28113_gb300 import sharded
from paper_2608_28113_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def dev():
    return torch.device("cuda", 0)


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()


def test_rank_order_sum_of_token_shares():
    n, chunk, chunks = 1040, 1536, 6
    a = wl.channel_magnitudes(n, 1.0, 8, 50.0, 51)
    xs = [wl.activation_chunk(chunk, a, 52, c) for c in range(chunks)]
    xd = [x.to(dev()) for x in xs]
    h_one = torch.zeros(n, device=dev())
    for x in xd:
        hs.hscale_hessian_diag_accumulate(x, h_one)
    for world in (2, 3, 4):
        parts = torch.zeros(world, n, device=dev())
        for r in range(world):
            c0, c1 = sharded.shard_range(chunks, r, world)
            for x in xd[c0:c1]:
                hs.hscale_hessian_diag_accumulate(x, parts[r])
        h1 = torch.empty(n, device=dev())
        h2 = torch.empty(n, device=dev())
        hs.hscale_hessian_sum_partials(parts, h1)
        hs.hscale_hessian_sum_partials(parts, h2)
        torch.cuda.synchronize()
        assert torch.equal(h1, h2)
        ref = parts[0].clone()
        for r in range(1, world):
            ref = ref + parts[r]
        assert torch.equal(h1, ref)                     # fp32 adds in rank order
        assert torch.all((h1 - h_one).abs() <= 1e-4 * h_one)
    h_ref = np.zeros(n)
    for x in xs:
        oracle.hessian_accumulate(wl.bf16_bits(x), h_ref)
    assert np.all(np.abs(h1.cpu().double().numpy() - h_ref) <= 1e-4 * h_ref)
    assert hs.hscale_device_error_flags() == 0


def rtn_sg(w):
    sg = torch.empty(1, device=dev())
    ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=dev())
    hs.hscale_rtn_scales(w, sg, None, ws)
    return sg


@pytest.mark.parametrize("kind", ["layer", "zero", "ties", "outlier_in_last_rows"])
def test_amax_word_all_reduced_gives_the_global_scale(kind):
    m, n = 96, 512
    if kind == "zero":
        w = torch.zeros(m, n, dtype=torch.bfloat16)
    elif kind == "ties":
        w = torch.full((m, n), 2688 * 2.0 ** -10, dtype=torch.float32).to(torch.bfloat16)
    else:
        w = wl.weight(m, n, 0.02, seed=61)
        if kind == "outlier_in_last_rows":
            w[m - 1, 7] = -37.5
    wd = w.to(dev())
    full = rtn_sg(wd)
    for world in (1, 2, 3, 5):
        words = []
        for r in range(world):
            r0, r1 = sharded.shard_range(m, r, world)
            b = torch.empty(1, dtype=torch.int32, device=dev())
            hs.hscale_amax_bits(wd[r0:r1].contiguous(), b)
            words.append(b)
        word = torch.stack(words).max(dim=0).values
        sg = torch.empty(1, device=dev())
        hs.hscale_global_scale_from_amax(word, sg)
        torch.cuda.synchronize()
        assert sg.cpu().numpy().tobytes() == full.cpu().numpy().tobytes()
    empty = torch.empty(0, n, dtype=torch.bfloat16, device=dev())
    b = torch.full((1,), 12345, dtype=torch.int32, device=dev())
    hs.hscale_amax_bits(empty, b)
    sg = torch.empty(1, device=dev())
    hs.hscale_global_scale_from_amax(b, sg)
    torch.cuda.synchronize()
    assert int(b.item()) == 0 and float(sg.item()) == 1.0


def test_row_shards_give_the_whole_matrix_search_bytes():
    m, n = 200, 1024
    w = wl.weight(m, n, 0.02, seed=71).to(dev())
    a = wl.channel_magnitudes(n, 1.0, 8, 50.0, 72)
    h = torch.zeros(n, device=dev())
    hs.hscale_hessian_diag_accumulate(wl.activation_chunk(2048, a, 72, 0).to(dev()), h)
    sg = rtn_sg(w)
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=dev())
    packed = torch.empty(m, n // 2, dtype=torch.uint8, device=dev())
    hs.hscale_refine_scales(w, h, sg, None, 4, 4, codes, packed)
    for world in (2, 3):
        for r in range(world):
            r0, r1 = sharded.shard_range(m, r, world)
            c, p = sharded.search_rows(w[r0:r1].contiguous(), h, sg, 4, 4)
            torch.cuda.synchronize()
            assert torch.equal(c, codes[r0:r1]) and torch.equal(p, packed[r0:r1])


def test_one_rank_sharded_layer_is_the_plain_path():
    m, n = 64, 512
    w = wl.weight(m, n, 0.02, seed=81).to(dev())
    a = wl.channel_magnitudes(n, 1.0, 8, 50.0, 82)
    xs = [wl.activation_chunk(1024, a, 82, c).to(dev()) for c in range(2)]
    h, sg, codes, packed = sharded.quantize_layer_sharded(xs, w, 4, 4)
    h0 = torch.zeros(n, device=dev())
    for x in xs:
        hs.hscale_hessian_diag_accumulate(x, h0)
    sg0 = rtn_sg(w)
    c0 = torch.empty_like(codes)
    p0 = torch.empty_like(packed)
    hs.hscale_refine_scales(w, h0, sg0, None, 4, 4, c0, p0)
    torch.cuda.synchronize()
    assert torch.equal(h, h0) and torch.equal(sg, sg0)
    assert torch.equal(codes, c0) and torch.equal(packed, p0)
