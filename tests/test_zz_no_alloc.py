"""The allocation-free apply entry point, salt_lora_apply_static.

Some callers cannot allocate device memory at the moment they apply: a
serving engine that plans all of its device memory before serving starts and
forbids allocations afterwards, or code running where cudaMalloc is not
allowed.  For them the library offers salt_lora_apply_static, which keeps the
intermediate V tiles in a static device array instead of the segments
object's workspace.

This file checks, through the C ABI, that two calls in a row give the same
result as the regular salt_lora_apply on the same inputs (within the parity
tolerance the other tests use), and that a batch too large for the static
array is refused before any device work.  Its name makes pytest collect it
last.
"""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


def test_static_apply_matches_regular_apply_twice(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config3()  # one Llama-3.1-8B layer: 256 tokens, 8 rank-64 centroids, Zipf users
    w.y_mode = "normal"
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        for l in (0, 1, 6):  # q 4096->4096, k 4096->1024, down 14336->4096
            x = bf16_tensor(w.x(l))
            y0 = w.y_in(l)
            y_reg = bf16_tensor(y0)
            salt.salt_lora_apply(r.ctx, r.seg, l, x, y_reg)
            torch.cuda.synchronize()
            ref = wl.bf16_bits_to_float(bf16_bits(y_reg)).astype(np.float64)
            for call in range(2):
                y = bf16_tensor(y0)
                salt.salt_lora_apply_static(r.ctx, r.seg, l, x, y)
                torch.cuda.synchronize()
                assert_close(bf16_bits(y), ref, f"static apply, layer {l}, call {call}")
        assert r.device_error() == 0


def test_static_apply_refuses_batches_beyond_its_scratch(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner
    salt = salt_lib
    T = 16384  # 8 domains of 2048 tokens: far more than 64 row blocks of <= 128 tokens
    slot = (np.arange(T) % 64).astype(np.int32)
    w = wl.Workload("many_blocks", 11, [("p", 64, 64)], 8, [8] * 8, 64, [1] * 64,
                    dom_ids=slot % 8, slot_ids=slot)
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        x = torch.zeros(T, 64, dtype=torch.bfloat16, device="cuda")
        y = torch.zeros(T, 64, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply_static(r.ctx, r.seg, 0, x, y)
        assert e.value.name == "SALT_ERR_TOO_MANY_TOKENS"
        torch.cuda.synchronize()
        assert (y == 0).all()
