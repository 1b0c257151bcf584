"""Failure detection on the GPU without a fault.

Every wait inside the path's kernels is bounded: when an mbarrier phase does
not complete in time, the wait records PIC_DEV_TIMEOUT in the device status
word and the kernel returns instead of hanging.  pic_wait_probe runs that
same bounded wait in a one-warp kernel, on a barrier that something arrives
on (the wait completes) or that nothing arrives on (the wait runs out after
the given limit).  The tests read the status the host sees and check that
the context keeps running work afterwards.
"""
import time

import pytest
import torch

pytestmark = pytest.mark.gpu

PIC_DEV_TIMEOUT = 8


def test_wait_that_completes_reports_nothing(cuda_lib):
    pic = cuda_lib
    pic.pic_device_status()  # start from a clear status word
    pic.pic_wait_probe(True, 50_000_000)
    assert pic.pic_device_status() == (0, 0)


def test_wait_that_runs_out_reports_a_timeout_and_the_context_survives(cuda_lib):
    pic = cuda_lib
    pic.pic_device_status()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    pic.pic_wait_probe(False, 20_000_000)  # 20 ms, nothing arrives
    code, detail = pic.pic_device_status()
    elapsed = time.perf_counter() - t0
    assert (code, detail) == (PIC_DEV_TIMEOUT, -1)
    assert elapsed >= 0.02
    # the status word was cleared by the read, and the context still runs work
    assert pic.pic_device_status() == (0, 0)
    pic.pic_wait_probe(True, 50_000_000)
    assert pic.pic_device_status() == (0, 0)
    x = torch.arange(1024, device="cuda", dtype=torch.float32)
    assert float(x.sum()) == 1024 * 1023 / 2


def test_first_failure_is_kept_until_read(cuda_lib):
    pic = cuda_lib
    pic.pic_device_status()
    pic.pic_wait_probe(False, 1_000_000)
    pic.pic_wait_probe(True, 1_000_000)  # a later success does not clear it
    assert pic.pic_device_status()[0] == PIC_DEV_TIMEOUT
