"""The allocation-free score + select + compaction entry point.

Some callers cannot allocate device memory while they run: serving loops that
reserve their whole budget up front, latency-critical code that must avoid the
allocator's locks and synchronisation, and hosts whose framework owns every
device allocation.  zsaa_score_select_noalloc keeps its score scratch in a
fixed array the library holds instead of taking it from the memory pool.
These tests call it through the C ABI and compare it with the allocating
zsaa_score_select on the same inputs -- two calls in a row on different
inputs, so scratch left over from the first call would show in the second --
and check that sizes beyond the fixed array are refused before any work.
"""

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
