"""pic_copy_async: host <-> device copies by the library's copy kernel, bit for
bit, over ragged sizes, unaligned starts (copy-engine fallback) and both
directions; pageable and overlapping arguments are refused."""
import ctypes

import pytest
import torch

pytestmark = pytest.mark.gpu

SIZES = [1, 15, 16, 17, 4096 + 3, 1 << 20, 2361856 + 5]


def _bytes(n, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(0, 256, (n,), dtype=torch.uint8, generator=g)


@pytest.mark.parametrize("n", SIZES)
def test_host_to_device_and_back(cuda_lib, n):
    import paper_2607_28069_gb300 as pic
    src = _bytes(n, n).pin_memory()
    dev = torch.full((n,), 7, dtype=torch.uint8, device="cuda")
    pic.pic_copy_async(dev, src)
    back = torch.zeros(n, dtype=torch.uint8).pin_memory()
    pic.pic_copy_async(back, dev)
    torch.cuda.synchronize()
    assert torch.equal(dev.cpu(), src)
    assert torch.equal(back, src)


@pytest.mark.parametrize("n", [33, 1 << 16])
def test_device_to_device(cuda_lib, n):
    import paper_2607_28069_gb300 as pic
    a = _bytes(n, 3).cuda()
    b = torch.zeros_like(a)
    pic.pic_copy_async(b, a)
    torch.cuda.synchronize()
    assert torch.equal(a, b)


@pytest.mark.parametrize("offset", [1, 3, 8])
def test_unaligned_start_falls_back_and_stays_exact(cuda_lib, offset):
    import paper_2607_28069_gb300 as pic
    n = 5000
    src = _bytes(n + offset, 11).pin_memory()
    dev = torch.zeros(n + 16, dtype=torch.uint8, device="cuda")
    pic.pic_copy_async(dev[offset:offset + n], src[offset:])
    torch.cuda.synchronize()
    assert torch.equal(dev[offset:offset + n].cpu(), src[offset:])
    assert int(dev[:offset].sum()) == 0 and int(dev[offset + n:].sum()) == 0


def test_copy_is_stream_ordered(cuda_lib):
    """Upload, device work, download on one stream: the download sees the work."""
    import paper_2607_28069_gb300 as pic
    n = 1 << 20
    src = _bytes(n, 5).pin_memory()
    dev = torch.empty(n, dtype=torch.uint8, device="cuda")
    out = torch.empty(n, dtype=torch.uint8).pin_memory()
    pic.pic_copy_async(dev, src)
    dev.add_(1)
    pic.pic_copy_async(out, dev)
    torch.cuda.synchronize()
    assert torch.equal(out, src + 1)


def test_pageable_and_overlapping_arguments_refused(cuda_lib):
    import paper_2607_28069_gb300 as pic
    lib = pic.load()
    pageable = torch.zeros(4096, dtype=torch.uint8)   # not page-locked
    dev = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    st = lib.pic_copy_async(ctypes.c_void_p(dev.data_ptr()), ctypes.c_void_p(pageable.data_ptr()),
                            4096, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 1 and b"page-locked" in lib.pic_last_error()
    st = lib.pic_copy_async(ctypes.c_void_p(dev.data_ptr() + 16), ctypes.c_void_p(dev.data_ptr()),
                            64, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == 1 and b"overlapping" in lib.pic_last_error()
    assert lib.pic_copy_async(None, None, 0, None) == 0       # nothing to copy
