"""Residual swap-in (Section "Multi-Tenant Serving": only the residual moves
host -> device): ordering against applies, stale segments, blob checks."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, oracle_tables

pytestmark = pytest.mark.gpu


def _workload(wl):
    T = 48
    u = (wl.uniform(31, 1, T) * 6).astype(np.int32)
    return wl.Workload("swap", 31, [("p", 256, 384)], 2, [16, 16], 8, [2] * 8, dom_ids=u % 2, slot_ids=u)


def _oracle(oracle_mod, w, version_of):
    cents, res = oracle_tables(w, 0, version=version_of)
    return oracle_mod.apply(w.x(0), w.y_in(0), w.dom_ids, w.slot_ids, cents, res)


def test_reload_between_batches_on_side_stream(salt_lib, oracle_mod, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = _workload(wl)
    side = torch.cuda.Stream()
    comp = torch.cuda.Stream()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        x = bf16_tensor(w.x(0))
        y1 = bf16_tensor(w.y_in(0))
        y2 = bf16_tensor(w.y_in(0))
        r.build(stream=comp)
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y1, comp)
        # swap new residuals into slots 1 and 3 while the first apply may still run
        b1 = r.make_blob(1, version=7)
        b3 = r.make_blob(3, version=7)
        salt.salt_residual_load(r.ctx, 1, b1, side)
        salt.salt_residual_load(r.ctx, 3, b3, side)
        with pytest.raises(salt.SaltError) as e:  # the built batch names slots 1 and 3
            salt.salt_lora_apply(r.ctx, r.seg, 0, x, y2, comp)
        assert e.value.name == "SALT_ERR_STALE_SEGMENTS"
        r.build(stream=comp)  # waits for the swaps of the slots it names
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y2, comp)
        torch.cuda.synchronize()
        assert r.device_error() == 0
        got1, got2 = bf16_bits(y1), bf16_bits(y2)
    assert_close(got1, _oracle(oracle_mod, w, lambda u: 0), "before the swap")
    assert_close(got2, _oracle(oracle_mod, w, lambda u: 7 if u in (1, 3) else 0), "after the swap")


def test_unreferenced_slot_load_keeps_segments_valid(salt_lib, oracle_mod, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = _workload(wl)
    w.slot_ids = np.where(w.slot_ids == 7, 6, w.slot_ids).astype(np.int32)  # slot 7 unused
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        salt.salt_residual_load(r.ctx, 7, r.make_blob(7, version=3), torch.cuda.Stream())
        x = bf16_tensor(w.x(0))
        y = bf16_tensor(w.y_in(0))
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y)  # no stale error: slot 7 is not named
        torch.cuda.synchronize()
        got = bf16_bits(y)
    assert_close(got, _oracle(oracle_mod, w, lambda u: 0), "unrelated swap")


def test_apply_on_another_stream_waits_for_the_build(salt_lib, oracle_mod, wl):
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = _workload(wl)
    s_build, s_apply = torch.cuda.Stream(), torch.cuda.Stream()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        x = bf16_tensor(w.x(0))
        y = bf16_tensor(w.y_in(0))
        torch.cuda.synchronize()
        r.build(stream=s_build)
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y, s_apply)
        torch.cuda.synchronize()
        got = bf16_bits(y)
    assert_close(got, _oracle(oracle_mod, w, lambda u: 0), "cross-stream")


def test_blob_checks(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner
    salt = salt_lib
    w = _workload(wl)
    with SaltRunner(w) as r:
        good = r.make_blob(0)
        # pageable host memory is refused
        with pytest.raises(salt.SaltError) as e:
            salt.salt_residual_load(r.ctx, 0, good.numpy().copy(), None)
        assert e.value.name == "SALT_ERR_NOT_PINNED_HOST"
        # wrong magic
        bad = good.clone().pin_memory()
        bad[0] ^= 0xFF
        with pytest.raises(salt.SaltError) as e:
            salt.salt_residual_load(r.ctx, 0, bad, None)
        assert e.value.name == "SALT_ERR_BAD_BLOB"
        # a blob packed for another layer table
        other = torch.empty(salt.salt_residual_blob_bytes([256], [392], 2), dtype=torch.uint8, pin_memory=True)
        salt.salt_residual_blob_pack([256], [392], 2, 1.0, np.zeros(512, np.uint16), np.zeros(784, np.uint16),
                                     other.numpy(), other.numel())
        with pytest.raises(salt.SaltError) as e:
            salt.salt_residual_load(r.ctx, 0, other, None)
        assert e.value.name == "SALT_ERR_BAD_BLOB"
        # rank above the context's r_max (2)
        big = r.make_blob(0, rank=3)
        with pytest.raises(salt.SaltError) as e:
            salt.salt_residual_load(r.ctx, 0, big, None)
        assert e.value.name == "SALT_ERR_RANK"
        with pytest.raises(salt.SaltError) as e:
            salt.salt_residual_load(r.ctx, 8, good, None)
        assert e.value.name == "SALT_ERR_SLOT_RANGE"


def test_huge_page_host_blob_swap(salt_lib, oracle_mod, wl):
    # salt_host_alloc memory is page-locked: a blob packed into it swaps in
    # asynchronously and the apply reads the new residual.
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = _workload(wl)
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        nb = r.blob_bytes(2)
        hb = salt.salt_host_alloc(3 * nb + 1000)
        try:
            assert hb.nbytes == 3 * nb + 1000 and int(hb.tensor[:4096].sum()) == 0
            blob = hb.tensor[nb:2 * nb]
            r.make_blob(2, version=5, out=blob)
            side = torch.cuda.Stream()
            salt.salt_residual_load(r.ctx, 2, blob, side)
            r.build()
            x = bf16_tensor(w.x(0))
            y = bf16_tensor(w.y_in(0))
            salt.salt_lora_apply(r.ctx, r.seg, 0, x, y)
            torch.cuda.synchronize()
            got = bf16_bits(y)
        finally:
            hb.close()
    assert_close(got, _oracle(oracle_mod, w, lambda u: 5 if u == 2 else 0), "huge-page host blob")


def test_batch_load_between_batches_on_side_stream(salt_lib, oracle_mod, wl):
    """salt_residual_load_batch: the same ordering as single loads (the swap
    waits for the applies that read the slots, the segments turn stale, a
    rebuild waits for the copies), one call for several slots; a bad blob in
    the batch loads nothing."""
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = _workload(wl)
    side = torch.cuda.Stream()
    comp = torch.cuda.Stream()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        x = bf16_tensor(w.x(0))
        y1 = bf16_tensor(w.y_in(0))
        y2 = bf16_tensor(w.y_in(0))
        y3 = bf16_tensor(w.y_in(0))
        r.build(stream=comp)
        salt.salt_lora_apply(r.ctx, r.seg, 0, x, y1, comp)
        # one blob from a huge-page region of the library, two from torch's pinned memory
        nb = r.blob_bytes(2)
        region = salt.salt_host_alloc(nb)
        try:
            b0 = r.make_blob(0, version=5, out=region.tensor[:nb])
            b2 = r.make_blob(2, version=5)
            b5 = r.make_blob(5, version=5)
            # a batch holding one bad blob is refused before anything is enqueued
            bad = r.make_blob(4, version=5).clone().pin_memory()
            bad[0] ^= 0xFF  # magic
            with pytest.raises(salt.SaltError):
                salt.salt_residual_load_batch(r.ctx, [0, 4], [b0, bad], side)
            salt.salt_lora_apply(r.ctx, r.seg, 0, x, y2, comp)  # still valid: nothing was loaded
            salt.salt_residual_load_batch(r.ctx, [0, 2, 5], [b0, b2, b5], side)
            with pytest.raises(salt.SaltError) as e:
                salt.salt_lora_apply(r.ctx, r.seg, 0, x, y3, comp)
            assert e.value.name == "SALT_ERR_STALE_SEGMENTS"
            r.build(stream=comp)
            salt.salt_lora_apply(r.ctx, r.seg, 0, x, y3, comp)
            torch.cuda.synchronize()
            assert r.device_error() == 0
            got1, got2, got3 = bf16_bits(y1), bf16_bits(y2), bf16_bits(y3)
        finally:
            torch.cuda.synchronize()
            salt.salt_host_free(region)
    assert_close(got1, _oracle(oracle_mod, w, lambda u: 0), "before the batch")
    assert_close(got2, _oracle(oracle_mod, w, lambda u: 0), "after the refused batch")
    assert_close(got3, _oracle(oracle_mod, w, lambda u: 5 if u in (0, 2, 5) else 0), "after the batch")
