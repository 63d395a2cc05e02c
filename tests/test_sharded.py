"""Sharding of the hot path across ranks (calibration tokens for h, rows of W for the search), tested on CPU with gloo ranks.

The orchestration in paper_2608_28113_gb300.sharded -- token shares for the Hessian pass,
the all-gather of the partials and their rank-order sum, the all-reduce with MAX of the amax
word, the row shares of the search -- runs here with world sizes 2 and 3 on the gloo backend.
The per-rank compute is the fp64 CPU oracle behind the same backend interface the CUDA
library implements (the GPU side of the interface is tested in test_gpu_sharded.py):

* the sharded h is within 1e-4 of the oracle's one-rank h over every token, the same bits on
  every rank, and the same bits on a second run;
* s_g equals the oracle's global scale of the whole matrix;
* every rank's codes and nibbles equal, byte for byte, the one-rank search of its rows with
  the same fp32 h and s_g.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_28113_gb300.sharded import shard_range  # noqa: E402

M, N, CHUNK, CHUNKS, DOWN, UP = 96, 256, 384, 5, 4, 4


def free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def layer():
    from paper_2608_28113_gb300 import workloads as wl
    w = wl.weight(M, N, 0.02, seed=41)
    a = wl.channel_magnitudes(N, 1.0, 8, 50.0, 42)
    xs = [wl.activation_chunk(CHUNK, a, 43, c) for c in range(CHUNKS)]
    return w, xs


class OracleBackend:
    """The per-rank steps of paper_2608_28113_gb300.sharded on the fp64 CPU oracle."""

    def __init__(self):
        import oracle
        from paper_2608_28113_gb300 import workloads as wl
        oracle.set_threads(1)
        self.o, self.wl = oracle, wl

    def hessian_partial(self, chunks, n, device):
        h = np.zeros(n)
        for x in chunks:
            self.o.hessian_accumulate(self.wl.bf16_bits(x), h)
        return torch.from_numpy(h.astype(np.float32))

    def sum_partials(self, partials):
        s = partials[0].clone()
        for r in range(1, partials.shape[0]):
            s = s + partials[r]          # fp32 round-to-nearest adds in rank order
        return s

    def amax_bits(self, w):
        b = self.wl.bf16_bits(w).astype(np.int64) & 0x7FFF
        return torch.tensor([int(b.max()) if b.size else 0], dtype=torch.int32)

    def global_scale(self, bits):
        word = np.full((1, 16), int(bits[0]), dtype=np.uint16)
        s_g, _ = self.o.global_scale(word)
        return torch.tensor([s_g], dtype=torch.float32)

    def search(self, w, h, sg, down, up):
        ref = self.o.refine(self.wl.bf16_bits(w), h.numpy(), float(sg[0]), None, down, up)
        return torch.from_numpy(ref["codes"]), torch.from_numpy(ref["packed"])


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    from paper_2608_28113_gb300 import sharded
    dist.init_process_group("gloo")
    try:
        w, xs = layer()
        c0, c1 = shard_range(CHUNKS, rank, world)
        r0, r1 = shard_range(M, rank, world)
        backend = OracleBackend()
        runs = []
        for _ in range(2):
            h, sg, codes, packed = sharded.quantize_layer_sharded(xs[c0:c1], w[r0:r1].contiguous(), DOWN, UP,
                                                                  backend=backend)
            runs.append((h.numpy().tobytes(), float(sg[0]), codes.numpy().tobytes(), packed.numpy().tobytes()))
        out[rank] = {"runs": runs, "rows": (r0, r1)}
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_token_and_row_shards_give_the_one_rank_results(world):
    import oracle
    from paper_2608_28113_gb300 import workloads as wl
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_rank, args=(world, free_port(), out), nprocs=world, join=True)
    w, xs = layer()
    wb = wl.bf16_bits(w)
    h_ref = np.zeros(N)
    for x in xs:
        oracle.hessian_accumulate(wl.bf16_bits(x), h_ref)
    s_ref, _ = oracle.global_scale(wb)
    h0 = out[0]["runs"][0][0]
    for r in range(world):
        runs = out[r]["runs"]
        assert runs[0] == runs[1]                       # deterministic
        assert runs[0][0] == h0                         # the same h on every rank
        assert np.float32(runs[0][1]) == np.float32(s_ref)
    h = np.frombuffer(h0, dtype=np.float32)
    assert np.all(np.abs(h - h_ref) <= 1e-4 * h_ref)
    ref = oracle.refine(wb, h, s_ref, None, DOWN, UP)   # the one-rank search, the same h and s_g
    rows = 0
    for r in range(world):
        r0, r1 = out[r]["rows"]
        codes = np.frombuffer(out[r]["runs"][0][2], dtype=np.uint8).reshape(r1 - r0, N // 16)
        packed = np.frombuffer(out[r]["runs"][0][3], dtype=np.uint8).reshape(r1 - r0, N // 2)
        assert np.array_equal(codes, ref["codes"][r0:r1])
        assert np.array_equal(packed, ref["packed"][r0:r1])
        rows += r1 - r0
    assert rows == M


def test_shard_ranges_cover_the_items_in_order():
    for total, world, align in ((0, 2, 1), (7, 3, 1), (96, 5, 1), (262144, 8, 8192), (10000, 3, 4096), (5, 8, 1)):
        prev = 0
        for r in range(world):
            a, b = shard_range(total, r, world, align)
            assert a == prev and a <= b
            assert a % align == 0
            prev = b
        assert prev == total
    with pytest.raises(ValueError):
        shard_range(10, 2, 2)
