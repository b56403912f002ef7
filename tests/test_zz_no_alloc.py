"""The allocation-free score + select + compaction entry point.

Some callers cannot allocate device memory while they run: serving loops that
reserve their whole budget up front, latency-critical code that must avoid the
allocator's locks and synchronisation, and hosts whose framework owns every
device allocation.  zsaa_score_select_noalloc keeps its score scratch in a
fixed array the library holds instead of taking it from the memory pool.
These tests call it through the C ABI and compare it with the allocating
zsaa_score_select on the same inputs -- two calls in a row on different
inputs, so scratch left over from the first call would show in the second --
check that sizes beyond the fixed array are refused before any work, and that
a call really allocates nothing: neither from the device's stream-ordered
memory pool (whose high-water mark of used memory stays at zero across the
call, while the allocating entry point raises it) nor with a plain device
allocation (the free device memory is unchanged).
"""

import ctypes

import pytest
import torch

from paper_2509_01190_gb300 import inputs as I
from tests.helpers import need_gpu

pytestmark = pytest.mark.gpu


def test_noalloc_matches_allocating_entry_point_on_two_calls(zlib):
    need_gpu()
    z = zlib
    for B, L, d, k, seed in [(4, 1000, 512, 300, 21), (3, 4096, 256, 1024, 22)]:
        hidden = I.make_hidden(B, L, d, seed=seed, device="cuda")
        ref_idx = torch.empty(B, k, device="cuda", dtype=torch.int32)
        ref_rows = torch.empty(B, k, d, device="cuda", dtype=torch.bfloat16)
        z.zsaa_score_select(hidden, B, L, d, k, ref_idx, ref_rows)
        idx = torch.full((B, k), -1, device="cuda", dtype=torch.int32)
        rows = torch.zeros(B, k, d, device="cuda", dtype=torch.bfloat16)
        z.zsaa_score_select_noalloc(hidden, B, L, d, k, idx, rows)
        torch.cuda.synchronize()
        # same kernels on the same inputs: indices and rows identical
        assert torch.equal(idx, ref_idx)
        assert torch.equal(rows.view(torch.int16), ref_rows.view(torch.int16))
    z.zsaa_device_status()


def test_noalloc_refuses_sizes_beyond_its_scratch(zlib):
    need_gpu()
    fake = 1 << 20  # never dereferenced: the size check comes first
    with pytest.raises(zlib.ZsaaError) as e:
        zlib.zsaa_score_select_noalloc(fake, 2, 1 << 20, 8, 5, fake, None, stream=0)
    assert e.value.status == zlib.ZSAA_ERR_INVALID_ARG
    assert "fixed scratch" in zlib.zsaa_last_error()


CU_MEMPOOL_ATTR_USED_MEM_HIGH = 8  # CUmemPool_attribute, cuda.h


def _pool_used_high():
    """(read, reset) of the default memory pool's high-water mark of used
    bytes on the current device, through the driver API."""
    cu = ctypes.CDLL("libcuda.so.1")
    dev, pool = ctypes.c_int(), ctypes.c_void_p()
    assert cu.cuCtxGetDevice(ctypes.byref(dev)) == 0
    assert cu.cuDeviceGetDefaultMemPool(ctypes.byref(pool), dev) == 0

    def read():
        v = ctypes.c_uint64()
        assert cu.cuMemPoolGetAttribute(pool, CU_MEMPOOL_ATTR_USED_MEM_HIGH, ctypes.byref(v)) == 0
        return v.value

    def reset():
        v = ctypes.c_uint64(0)
        assert cu.cuMemPoolSetAttribute(pool, CU_MEMPOOL_ATTR_USED_MEM_HIGH, ctypes.byref(v)) == 0
    return read, reset


def test_noalloc_call_allocates_nothing(zlib):
    need_gpu()
    z = zlib
    torch.cuda.init()
    # one call first, so that lazily loaded kernels are resident
    B, L, d, k = 2, 512, 256, 100
    h0 = I.make_hidden(B, L, d, seed=31, device="cuda")
    i0 = torch.empty(B, k, device="cuda", dtype=torch.int32)
    r0 = torch.empty(B, k, d, device="cuda", dtype=torch.bfloat16)
    z.zsaa_score_select_noalloc(h0, B, L, d, k, i0, r0)
    z.zsaa_score_select(h0, B, L, d, k, i0, r0)
    torch.cuda.synchronize()
    # then a size not seen before, with every tensor made up front
    B, L, d, k = 5, 3000, 384, 700
    hidden = I.make_hidden(B, L, d, seed=32, device="cuda")
    idx = torch.empty(B, k, device="cuda", dtype=torch.int32)
    rows = torch.empty(B, k, d, device="cuda", dtype=torch.bfloat16)
    torch.cuda.synchronize()
    read, reset = _pool_used_high()
    # control: the allocating entry point takes its scores from the pool
    reset()
    z.zsaa_score_select(hidden, B, L, d, k, idx, rows)
    torch.cuda.synchronize()
    assert read() >= 4 * B * L
    reset()
    free_before = torch.cuda.mem_get_info()[0]
    z.zsaa_score_select_noalloc(hidden, B, L, d, k, idx, rows)
    torch.cuda.synchronize()
    assert read() == 0
    assert torch.cuda.mem_get_info()[0] == free_before
    z.zsaa_device_status()
