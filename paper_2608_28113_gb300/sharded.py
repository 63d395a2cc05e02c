"""The hot path split across GPUs: one process per GPU, torch.distributed between them.

Both parts of the path split without any exchange inside a kernel:

* Hessian pass, calibration tokens split across ranks (h is a sum over tokens, Sec. 3.2,
  Eq. 4).  Each rank accumulates a partial h over the chunks of its token share, the partials
  are all-gathered (n fp32 per rank), and every rank adds them in rank order
  (hscale_hessian_sum_partials).  Every rank then holds the same h, bit for bit, on every run.
* Search, rows of W split across ranks (every group is searched on its own given h and the
  global scale, Algorithm 1).  The global scale needs the amax of the whole matrix (Sec. 3.3):
  each rank takes the amax word of its rows (hscale_amax_bits), one all-reduce with MAX on
  that int32 gives the word of the whole matrix, and every rank forms the same s_g
  (hscale_global_scale_from_amax).  A rank's codes and nibbles are then exactly the bytes a
  one-rank search writes for its rows.

The per-rank compute is a backend object; the default, `CudaBackend`, is the CUDA library
(device tensors, the current stream).  The orchestration here (the shares, the collectives and
their order) does no arithmetic of the method itself.  Without an initialised process group
the functions run as a single rank.
"""
from __future__ import annotations

import torch

__all__ = ["CudaBackend", "shard_range", "rank_and_world", "hessian_sharded", "global_scale_sharded",
           "search_rows", "quantize_layer_sharded"]


def rank_and_world(group=None) -> tuple[int, int]:
    """(rank, world size) of the process group, (0, 1) without one."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized():
        return dist.get_rank(group), dist.get_world_size(group)
    return 0, 1


def shard_range(total: int, rank: int, world: int, align: int = 1) -> tuple[int, int]:
    """This rank's contiguous share [start, stop) of `total` items, in whole units of `align`
    items (the last unit may be short), balanced to within one unit; shares of consecutive
    ranks are adjacent and together cover [0, total)."""
    if world < 1 or not 0 <= rank < world or align < 1 or total < 0:
        raise ValueError("need world >= 1, 0 <= rank < world, align >= 1, total >= 0")
    units = (total + align - 1) // align
    lo, hi = units * rank // world, units * (rank + 1) // world
    return min(lo * align, total), min(hi * align, total)


class CudaBackend:
    """The per-rank steps on the CUDA library."""

    def __init__(self):
        from . import (hscale_amax_bits, hscale_global_scale_from_amax, hscale_hessian_diag_accumulate,
                       hscale_hessian_sum_partials, hscale_refine_scales, load)
        load()
        self._acc, self._sum = hscale_hessian_diag_accumulate, hscale_hessian_sum_partials
        self._amax, self._sg, self._refine = hscale_amax_bits, hscale_global_scale_from_amax, hscale_refine_scales

    def hessian_partial(self, chunks, n: int, device) -> torch.Tensor:
        h = torch.zeros(n, dtype=torch.float32, device=device)
        for x in chunks:
            self._acc(x, h)
        return h

    def sum_partials(self, partials: torch.Tensor) -> torch.Tensor:
        h = torch.empty(partials.shape[1], dtype=torch.float32, device=partials.device)
        return self._sum(partials, h)

    def amax_bits(self, w: torch.Tensor) -> torch.Tensor:
        bits = torch.empty(1, dtype=torch.int32, device=w.device)
        return self._amax(w, bits)

    def global_scale(self, bits: torch.Tensor) -> torch.Tensor:
        sg = torch.empty(1, dtype=torch.float32, device=bits.device)
        self._sg(bits, sg)
        return sg

    def search(self, w: torch.Tensor, h: torch.Tensor, sg: torch.Tensor, down: int, up: int):
        m, n = w.shape
        codes = torch.empty(m, n // 16, dtype=torch.uint8, device=w.device)
        packed = torch.empty(m, n // 2, dtype=torch.uint8, device=w.device)
        if m:
            self._refine(w, h, sg, None, down, up, codes, packed)
        return codes, packed


def hessian_sharded(local_chunks, n: int, device=None, group=None, backend=None) -> torch.Tensor:
    """h over every rank's calibration tokens: this rank's partial over `local_chunks` (its
    token share, bf16 [tokens_i, n] each), all-gathered and summed in rank order."""
    import torch.distributed as dist
    backend = backend or CudaBackend()
    device = device if device is not None else (local_chunks[0].device if local_chunks else "cpu")
    partial = backend.hessian_partial(list(local_chunks), n, device)
    _, world = rank_and_world(group)
    if world == 1:
        return backend.sum_partials(partial.reshape(1, n))
    parts = [torch.empty_like(partial) for _ in range(world)]
    dist.all_gather(parts, partial, group=group)
    return backend.sum_partials(torch.stack(parts))


def global_scale_sharded(w_local: torch.Tensor, group=None, backend=None) -> torch.Tensor:
    """s_g of the whole matrix from this rank's rows: the amax words all-reduced with MAX."""
    import torch.distributed as dist
    backend = backend or CudaBackend()
    bits = backend.amax_bits(w_local)
    _, world = rank_and_world(group)
    if world > 1:
        dist.all_reduce(bits, op=dist.ReduceOp.MAX, group=group)
    return backend.global_scale(bits)


def search_rows(w_local: torch.Tensor, h: torch.Tensor, sg: torch.Tensor, down: int, up: int, backend=None):
    """Codes and packed nibbles of this rank's rows (no collective)."""
    backend = backend or CudaBackend()
    return backend.search(w_local, h, sg, down, up)


def quantize_layer_sharded(local_chunks, w_local: torch.Tensor, down: int, up: int, group=None, backend=None):
    """One layer across the ranks: h over every rank's tokens, s_g over every rank's rows, then
    the search of this rank's rows.  Returns (h, s_g, codes, packed); h and s_g are the same on
    every rank, codes and packed cover this rank's rows."""
    backend = backend or CudaBackend()
    n = w_local.shape[1]
    h = hessian_sharded(local_chunks, n, w_local.device, group, backend)
    sg = global_scale_sharded(w_local, group, backend)
    codes, packed = search_rows(w_local, h, sg, down, up, backend)
    return h, sg, codes, packed
