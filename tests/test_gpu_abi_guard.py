"""The library's device-buffer guard (include/rrq.h: rrq_check_buffer, the
check every entry point applies to each buffer before launching): a buffer
must lie, every byte of it, in device memory of the current device.  Freed
memory, a length that runs past the allocation, host memory and null are
refused; nothing here launches a kernel on a refused buffer."""
import ctypes

import pytest
import torch

from paper_2608_04048_gb300 import binding, build

pytestmark = pytest.mark.gpu

MiB = 1 << 20


@pytest.fixture(scope="module", autouse=True)
def lib():
    build.build()
    return binding.load_library()


def _segment_of(ptr: int):
    """(start, size) of the caching allocator's segment holding ptr."""
    for seg in torch.cuda.memory_snapshot():
        if seg["address"] <= ptr < seg["address"] + seg["total_size"]:
            return seg["address"], seg["total_size"]
    raise AssertionError("pointer outside every segment")


def test_device_tensor_accepted_whole_and_in_part():
    x = torch.empty(8 * MiB, dtype=torch.uint8, device="cuda")
    p = x.data_ptr()
    assert binding.rrq_check_buffer(p, x.numel()) == 0
    assert binding.rrq_check_buffer(p + 4096, 4096) == 0
    assert binding.rrq_check_buffer(p, 0) == 0  # the first byte only


def test_length_past_the_allocation_refused():
    x = torch.empty(64 * MiB, dtype=torch.uint8, device="cuda")
    start, size = _segment_of(x.data_ptr())
    end = start + size
    assert binding.rrq_check_buffer(start, size) == 0
    # far past the end: no run of device memory of that length exists
    assert binding.rrq_check_buffer(end - 16, 1 << 40) == 1
    # just past the end, when the byte after the segment is not device memory
    if binding.rrq_check_buffer(end, 1) != 0:
        assert binding.rrq_check_buffer(end - 16, 32) == 1


def test_freed_memory_refused():
    torch.cuda.synchronize()
    torch.cuda.empty_cache()
    # larger than every free block the allocator holds: a segment of its own
    free = [b["size"] for seg in torch.cuda.memory_snapshot() for b in seg["blocks"] if b["state"] == "inactive"]
    n = max([96 * MiB] + [f + 4 * MiB for f in free])
    x = torch.empty((n + 2 * MiB - 1) // (2 * MiB) * (2 * MiB), dtype=torch.uint8, device="cuda")
    p = x.data_ptr()
    assert _segment_of(p) == (p, x.numel())
    assert binding.rrq_check_buffer(p, x.numel()) == 0
    del x
    torch.cuda.synchronize()
    torch.cuda.empty_cache()  # the segment goes back to the driver
    assert binding.rrq_check_buffer(p, 16) == 1


def test_host_and_null_refused():
    h = torch.empty(4096, dtype=torch.uint8, pin_memory=True)
    assert binding.rrq_check_buffer(h.data_ptr(), 4096) == 1
    plain = (ctypes.c_uint8 * 4096)()
    assert binding.rrq_check_buffer(ctypes.addressof(plain), 4096) == 1
    assert binding.rrq_check_buffer(0, 16) == 1


def test_entry_point_refuses_a_host_input_before_launching(lib):
    """rrq_quantize through the C ABI with W in pinned host memory: refused
    (a kernel given it would still only read host memory)."""
    rows, cols = 8, 256
    W = torch.zeros((rows, cols), dtype=torch.bfloat16, pin_memory=True)
    pkg = binding.Package.empty(rows, cols, 128, 2)
    P = ctypes.c_void_p * 2
    rc = lib.rrq_quantize(W.data_ptr(), rows, cols, 128, 2, P(*[c.data_ptr() for c in pkg.codes]),
                          P(*[s.data_ptr() for s in pkg.scales]), P(*[z.data_ptr() for z in pkg.zeros]), None)
    assert rc == 1
    torch.cuda.synchronize()
    assert binding.rrq_get_device_status() == 0
