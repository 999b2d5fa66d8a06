"""zarya_copy: byte-exact transfers between pinned host memory and the device
(and device to device) done by a kernel, eager and inside a CUDA graph, and
the calls it refuses without launching anything."""
import ctypes

import pytest
import torch

pytestmark = pytest.mark.gpu

SIZES = [1, 15, 16, 17, 4096 + 3, 2 * 1024 * 1024 + 32, (1 << 24) + 5]


@pytest.fixture(scope="module")
def zb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2609_19868_gb300 import build
    from paper_2609_19868_gb300 import _binding as zb

    build.build()
    zb.load()
    zb.check_device_error()
    return zb


def _bytes(n, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(0, 256, (n,), dtype=torch.uint8, generator=g)


@pytest.mark.parametrize("n", SIZES)
def test_host_to_device_to_host_is_exact(zb, n):
    src = _bytes(n, n).pin_memory()
    dev = torch.full((n,), 7, dtype=torch.uint8, device="cuda")
    back = torch.zeros(n, dtype=torch.uint8).pin_memory()
    zb.copy(dev, src)
    zb.copy(back, dev)
    torch.cuda.synchronize()
    assert torch.equal(dev.cpu(), src)
    assert torch.equal(back, src)


@pytest.mark.parametrize("n", [17, 1 << 20])
def test_device_to_device_and_offsets(zb, n):
    a = _bytes(n + 64, 3).cuda()
    b = torch.zeros(n + 64, dtype=torch.uint8, device="cuda")
    zb.copy(b[32:32 + n], a[16:16 + n])            # 16-byte aligned interior ranges
    torch.cuda.synchronize()
    assert torch.equal(b[32:32 + n], a[16:16 + n])
    assert (b[:32] == 0).all() and (b[32 + n:] == 0).all()   # nothing written outside


def test_copies_in_a_cuda_graph_follow_the_host_buffer(zb):
    n = 2 * 1024 * 1024 + 32
    host_in = _bytes(n, 1).pin_memory()
    host_out = torch.zeros(n, dtype=torch.uint8).pin_memory()
    dev = torch.empty(n, dtype=torch.uint8, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        zb.copy(dev, host_in, s)
        zb.copy(host_out, dev, s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        zb.copy(dev, host_in, s)
        zb.copy(host_out, dev, s)
    host_in.copy_(_bytes(n, 2))                     # new inputs, same buffer
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(host_out, host_in)


def test_refused_calls_launch_nothing(zb):
    lib = zb.load()
    vp = ctypes.c_void_p
    d = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    h = torch.zeros(4096, dtype=torch.uint8).pin_memory()
    pageable = torch.zeros(4096, dtype=torch.uint8)
    base = d.data_ptr()
    assert lib.zarya_copy(vp(base + 4), vp(h.data_ptr()), 64, None) == zb.ERR_INVALID_ARG
    assert lib.zarya_copy(vp(base), vp(base + 1024), 2048, None) == zb.ERR_INVALID_ARG  # overlap
    assert lib.zarya_copy(vp(h.data_ptr()), vp(h.data_ptr() + 2048), 64, None) == \
        zb.ERR_INVALID_ARG                                                     # host to host
    assert lib.zarya_copy(vp(pageable.data_ptr()), vp(base), 64, None) == zb.ERR_INVALID_ARG
    with pytest.raises(TypeError):
        zb.copy(d, pageable)
    torch.cuda.synchronize()
    assert (d == 0).all()
    assert zb.check_device_error() == 0
