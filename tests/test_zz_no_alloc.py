"""The allocation-free apply entry point, salt_lora_apply_static.

Some callers cannot allocate device memory at the moment they apply: a
serving engine that plans all of its device memory before serving starts and
forbids allocations afterwards, or code running where cudaMalloc is not
allowed.  For them the library offers salt_lora_apply_static, which keeps the
intermediate V tiles in a static device array instead of the segments
object's workspace.

This file checks, through the C ABI, that two calls in a row match the fp64
oracle (within the parity tolerance the other tests use) and are bit for bit
equal to the regular salt_lora_apply on the same inputs; that two segments
objects of different sizes, applied alternately through the shared static
scratch and interleaved with regular applies on one stream, each match the
oracle; and that a batch too large for the static array is refused before
any device work.  Its name makes pytest collect it last.
"""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, oracle_tables

pytestmark = pytest.mark.gpu


def _oracle(oracle_mod, w, l, rows=None):
    cents, res = oracle_tables(w, l)
    dom = w.dom_ids if rows is None else w.dom_ids[rows]
    slot = w.slot_ids if rows is None else w.slot_ids[rows]
    return oracle_mod.apply(w.x(l, rows), w.y_in(l, rows), dom, slot, cents, res)


def test_static_apply_matches_regular_apply_twice(salt_lib, oracle_mod, wl):
    """Two calls in a row: each within the tolerance of the fp64 oracle, and
    bit for bit equal to salt_lora_apply on the same inputs (the same split
    of the shrink, a deterministic reduction)."""
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
            reg = bf16_bits(y_reg)
            ref = _oracle(oracle_mod, w, l)
            for call in range(2):
                y = bf16_tensor(y0)
                salt.salt_lora_apply_static(r.ctx, r.seg, l, x, y)
                torch.cuda.synchronize()
                got = bf16_bits(y)
                assert_close(got, ref, f"static apply vs oracle, layer {l}, call {call}")
                np.testing.assert_array_equal(got, reg, err_msg=f"static vs regular apply, layer {l}, call {call}")
        assert r.device_error() == 0


def test_static_apply_alternating_segments(salt_lib, oracle_mod, wl):
    """Two segments objects of different sizes (all 256 tokens of the layer,
    and 96 of them) share the one static scratch; their static applies
    alternate with regular applies on one stream, and every result is
    checked against the oracle.  Stale counters or a wrong launch parity in
    the shared scratch would show up here."""
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config3()
    w.y_mode = "normal"
    rows_b = np.unique((wl.uniform(3, 901, 128) * w.T).astype(np.int64) % w.T)[:96]
    stream = torch.cuda.Stream()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build(stream=stream)
        seg_b = salt.salt_segments_create(r.ctx)
        try:
            salt.salt_build_segments(r.ctx, seg_b, w.dom_ids[rows_b], w.slot_ids[rows_b], stream=stream)
            plan = []
            for l in (0, 3, 6):
                plan += [("static", r.seg, l, None), ("regular", r.seg, l, None),
                         ("static", seg_b, l, rows_b), ("regular", seg_b, l, rows_b), ("static", seg_b, l, rows_b)]
            outs = []
            with torch.cuda.stream(stream):
                for kind, seg, l, rows in plan:
                    x = bf16_tensor(w.x(l, rows))
                    y = bf16_tensor(w.y_in(l, rows))
                    fn = salt.salt_lora_apply_static if kind == "static" else salt.salt_lora_apply
                    fn(r.ctx, seg, l, x, y, stream)
                    outs.append((kind, l, rows, x, y))
            stream.synchronize()
            assert r.device_error() == 0
            assert salt.salt_guard_check(r.ctx, r.seg) == 0 and salt.salt_guard_check(r.ctx, seg_b) == 0
            refs = {}
            for kind, l, rows, x, y in outs:
                key = (l, None if rows is None else len(rows))
                if key not in refs:
                    refs[key] = _oracle(oracle_mod, w, l, rows)
                assert_close(bf16_bits(y), refs[key], f"{kind} apply, layer {l}, {key[1] or w.T} tokens")
        finally:
            salt.salt_segments_destroy(seg_b)


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
