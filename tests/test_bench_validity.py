"""bench.py refuses to report work the kernels flagged as incomplete: a
device error flag read at any checkpoint (a bounded wait that gave up, an id
the kernels rejected) makes the run invalid.  The binding is replaced by a
fake on the CPU; no GPU fault is involved."""
import bench


class _FakeSalt:
    def __init__(self, flags):
        self.flags = list(flags)

    def salt_get_device_error(self, ctx, stream=None):
        return self.flags.pop(0) if self.flags else 0


def test_clean_run_is_valid():
    d = bench.DeviceErrors(_FakeSalt([0, 0, 0]), ctx=1)
    for where in ("warmup", "timed", "end"):
        assert d.check(where) == 0
    assert d.valid
    assert d.summary() == {"valid": True, "device_error_flags": {}}


def test_timeout_flag_makes_the_run_invalid():
    d = bench.DeviceErrors(_FakeSalt([0, 0x20, 0]), ctx=1)
    for where in ("warmup", "timed", "end"):
        d.check(where)
    assert not d.valid
    s = d.summary()
    assert s["valid"] is False and s["device_error_flags"] == {"timed": "0x20"}


def test_huge_page_report_finds_the_mapping():
    """The swap's host-memory report reads the mapping that holds a pointer
    from /proc/self/smaps: its size, and the bytes backed by huge pages."""
    import ctypes
    import mmap
    n = 4 << 20
    m = mmap.mmap(-1, n)
    buf = (ctypes.c_char * n).from_buffer(m)
    size, huge = bench.huge_page_bytes(ctypes.addressof(buf))
    assert size is not None and size >= n
    assert huge is not None and 0 <= huge <= size
    del buf
    m.close()
    assert bench.huge_page_bytes(0) == (None, None)
