"""Page-locked staging memory from nexus_host_alloc: registered with the
driver, zero-filled, and asynchronous copies to and from it move the bytes
unchanged."""
import ctypes

import pytest
import torch

from paper_2608_20397_gb300 import nexus

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    return torch.device("cuda:0")


@pytest.mark.parametrize("shape", [(1,), (3, 1000), (48, 65536 + 7), (2, 1 << 22)])
def test_round_trip_through_staging(dev, shape):
    h_in = nexus.host_empty(shape, torch.bfloat16)
    h_out = nexus.host_empty(shape, torch.bfloat16)
    assert not h_in.view(torch.int16).any()                 # fresh pages are zero
    g = torch.Generator().manual_seed(1)
    h_in.copy_(torch.randn(shape, generator=g).to(torch.bfloat16))
    s = torch.cuda.Stream(device=dev)
    d = torch.empty(shape, dtype=torch.bfloat16, device=dev)
    with torch.cuda.stream(s):
        d.copy_(h_in, non_blocking=True)
        d.mul_(-1)
        h_out.copy_(d, non_blocking=True)
    s.synchronize()
    assert torch.equal(h_out.view(torch.int16), (-h_in).view(torch.int16))


def test_direct_alloc_and_free(dev):
    L = nexus.lib()
    p = ctypes.c_void_p()
    assert L.nexus_host_alloc(5000, ctypes.byref(p)) == nexus.OK and p.value
    assert p.value % 4096 == 0
    ctypes.memset(p.value, 7, 5000)
    # a size that maps to another length, or an address inside the mapping, is refused
    assert L.nexus_host_free(p, 1 << 30) == nexus.EINVAL
    assert L.nexus_host_free(ctypes.c_void_p(p.value + 4096), 100) == nexus.EINVAL
    assert ctypes.string_at(p.value, 1) == b"\x07"   # still mapped
    assert L.nexus_host_free(p, 5000) == nexus.OK
    assert L.nexus_host_free(p, 5000) == nexus.EINVAL   # already returned


def test_views_keep_the_mapping(dev):
    t = nexus.host_empty((1024, 128), torch.float32)
    v = t[10:20]
    del t
    v.fill_(2.5)
    d = v.to(dev, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(d.cpu(), torch.full((10, 128), 2.5))


def test_large_staging_region(dev):
    # 600 MB: rounded up to whole transparent huge pages where the host has them
    shape = (300, 1 << 20)
    h = nexus.host_empty(shape, torch.bfloat16)
    assert not h[::37].view(torch.int16).any()
    d = torch.randn(shape, device=dev).to(torch.bfloat16)
    h.copy_(d, non_blocking=True)
    back = torch.empty_like(d)
    back.copy_(h, non_blocking=True)
    torch.cuda.synchronize()
    assert torch.equal(back.view(torch.int16), d.view(torch.int16))


def test_group_of_staging_tensors(dev):
    """Tensors carved out of one mapping: 64 KiB-aligned, disjoint, each moving
    its own bytes."""
    specs = [((3, 7), torch.bfloat16), ((5000,), torch.float32), ((1,), torch.int8),
             ((48, 64, 40, 128), torch.bfloat16)]
    ts = nexus.host_empty_group(specs)
    assert [tuple(t.shape) for t in ts] == [s for s, _ in specs]
    assert [t.dtype for t in ts] == [d for _, d in specs]
    starts = [t.data_ptr() for t in ts]
    assert all(p % 65536 == 0 for p in starts)
    ends = [p + t.numel() * t.element_size() for p, t in zip(starts, ts)]
    assert all(ends[i] <= starts[i + 1] for i in range(len(ts) - 1))
    g = torch.Generator().manual_seed(3)
    for t in ts:
        t.copy_(torch.randint(-100, 100, t.shape, generator=g).to(t.dtype))
    want = [t.clone() for t in ts]
    d = [t.to(dev, non_blocking=True) for t in ts]
    torch.cuda.synchronize()                 # the copies have read the host bytes
    for t in ts:
        t.zero_()
    for t, x in zip(ts, d):
        t.copy_(x, non_blocking=True)
    torch.cuda.synchronize()
    assert all(torch.equal(t, w) for t, w in zip(ts, want))
    assert nexus.host_empty_group([]) == []
