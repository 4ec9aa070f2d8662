"""Failure detection on the GPU without a fault: a bounded wait that runs out
raises SALT_DEVERR_TIMEOUT, and the context keeps working afterwards."""
import time

import pytest
import torch

from gpu_helpers import assert_close, oracle_tables

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives(salt_lib, oracle_mod, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config0()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        assert r.device_error() == 0
        t0 = time.perf_counter()
        salt.salt_selftest_wait_timeout(r.ctx)
        flags = r.device_error()  # synchronises the stream
        waited = time.perf_counter() - t0
        assert flags & 0x20, hex(flags)  # SALT_DEVERR_TIMEOUT
        assert waited < 30.0
        assert r.device_error() == 0  # read and cleared
        # the context and the GPU are still usable: a normal apply is correct
        x = bf16_tensor(w.x(0))
        y = bf16_tensor(w.y_in(0))
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y)
        torch.cuda.synchronize()
        assert r.device_error() == 0
        got = bf16_bits(y)
    cents, res = oracle_tables(w, 0)
    assert_close(got, oracle_mod.apply(w.x(0), w.y_in(0), w.dom_ids, w.slot_ids, cents, res), "after the timeout")
