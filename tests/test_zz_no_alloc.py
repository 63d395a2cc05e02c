"""hscale_rtn_scales_noalloc, the entry point for callers that cannot allocate device
memory (for instance a plugin handed only its input and output tensors).

It must give exactly what hscale_rtn_scales gives with a caller-owned workspace, on two
calls in a row: the second call uses a matrix with a smaller maximum, so a scratch word
left over from the first call would show up as a wrong global scale.  The file is named
to be collected last; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

import paper_2608_28113_gb300 as hs
from paper_2608_28113_gb300 import workloads as wl

pytestmark = pytest.mark.gpu


def with_workspace(w):
    m, n = w.shape
    sg = torch.empty(1, dtype=torch.float32, device=w.device)
    codes = torch.empty(m, n // 16, dtype=torch.uint8, device=w.device)
    ws = torch.empty(hs.hscale_rtn_workspace_bytes(), dtype=torch.uint8, device=w.device)
    hs.hscale_rtn_scales(w, sg, codes, ws)
    return sg, codes


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()
    dev = torch.device("cuda", 0)
    first = wl.weight(512, 1024, 0.02, seed=21).to(dev)
    second = (wl.weight(256, 2048, 0.02, seed=22) * 0.25).to(dev)   # smaller amax than `first`
    assert second.abs().max() < first.abs().max()
    for w in (first, second):
        m, n = w.shape
        sg = torch.full((1,), -1.0, dtype=torch.float32, device=dev)
        codes = torch.full((m, n // 16), 255, dtype=torch.uint8, device=dev)
        hs.hscale_rtn_scales_noalloc(w, sg, codes)
        ref_sg, ref_codes = with_workspace(w)
        torch.cuda.synchronize()
        # bit-exact, the rule the parity tests apply to s_g and codes
        assert sg.cpu().numpy().tobytes() == ref_sg.cpu().numpy().tobytes()
        assert np.array_equal(codes.cpu().numpy(), ref_codes.cpu().numpy())
    assert hs.hscale_device_error_flags() == 0


def test_noalloc_allocates_no_device_memory():
    """After a first call (which resolves the scratch address and loads the kernels), further
    calls change neither torch's allocator nor the device's free memory."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()
    dev = torch.device("cuda", 0)
    w = wl.weight(512, 1024, 0.02, seed=23).to(dev)
    sg = torch.empty(1, dtype=torch.float32, device=dev)
    codes = torch.empty(512, 1024 // 16, dtype=torch.uint8, device=dev)
    hs.hscale_rtn_scales_noalloc(w, sg, codes)
    torch.cuda.synchronize()
    allocated = torch.cuda.memory_allocated(dev)
    free_before, _ = torch.cuda.mem_get_info(dev)
    for _ in range(3):
        hs.hscale_rtn_scales_noalloc(w, sg, codes)
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info(dev)
    assert torch.cuda.memory_allocated(dev) == allocated
    assert free_after == free_before
