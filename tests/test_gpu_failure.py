"""Failure detection on the GPU without a fault: a bounded wait that runs out.

The library's TMA pipelines bound every mbarrier wait; a wait that runs out sets a sticky
device flag and the kernel ends normally.  The self-test kernel drives that same path with
a small poll limit on an mbarrier that nothing arrives on, and the host reads the status;
afterwards the context must still run the hot path.
"""
import pytest
import torch

import paper_2608_28113_gb300 as hs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    hs.load()


def test_bounded_wait_runs_out_reports_and_the_context_survives():
    dev = torch.device("cuda", 0)
    hs.hscale_device_error_flags()                      # start from a clean state
    for polls in (0, 1000):
        hs.hscale_selftest_bounded_wait(polls)
        torch.cuda.synchronize()
        assert hs.hscale_device_error_flags() & 1, f"timeout not reported ({polls} polls)"
        assert hs.hscale_device_error_flags() == 0      # the flags clear on read
    x = torch.ones(256, 64, dtype=torch.bfloat16, device=dev) * 2
    h = torch.zeros(64, dtype=torch.float32, device=dev)
    hs.hscale_hessian_diag_accumulate(x, h)
    torch.cuda.synchronize()
    assert torch.all(h == 256 * 4.0)
    assert hs.hscale_device_error_flags() == 0
