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
