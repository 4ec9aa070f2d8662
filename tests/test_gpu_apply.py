"""salt_lora_apply on the GPU against the fp64 oracle, element by element."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, guarded_like, guards_intact, oracle_tables

pytestmark = pytest.mark.gpu


def run_gpu(wl, groups, y_mode=None, scales_c=None, repeat=1):
    """Pin, swap every slot, build, apply each group; return {layer: y bits}.
    Every y sits between guard bands, and the library's own guard bands
    (centroid arenas, slot pool, V tiles, split partials) are checked after
    the applies: a store past any of these buffers fails the test."""
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits
    if y_mode:
        wl.y_mode = y_mode
    out = {}
    with SaltRunner(wl) as r:
        r.pin_centroids(scales_c)
        r.load_slots()
        r.build()
        for grp in groups:
            xs, ys = r.alloc_xy(grp)
            gys = [guarded_like(y) for y in ys]
            ys = [g[0] for g in gys]
            for _ in range(repeat):
                r.apply(grp, xs, ys)
            torch.cuda.synchronize()
            for l, y, (_, buf) in zip(grp, ys, gys):
                out[l] = bf16_bits(y)
                assert guards_intact(buf), f"a store ran past y of layer {l}"
        torch.cuda.synchronize()
        assert r.device_error() == 0
        from paper_2608_03579_gb300 import salt
        assert salt.salt_guard_check(r.ctx, r.seg) == 0, "a guard band of the library's buffers changed"
    return out


def oracle_layer(oracle_mod, wl, l, rows=None, scales_c=None):
    cents, res = oracle_tables(wl, l, scales_c=scales_c)
    x = wl.x(l, rows)
    y = wl.y_in(l, rows)
    dom = wl.dom_ids if rows is None else wl.dom_ids[rows]
    slot = wl.slot_ids if rows is None else wl.slot_ids[rows]
    return oracle_mod.apply(x, y, dom, slot, cents, res)


@pytest.mark.parametrize("y_mode", ["zeros", "normal"])
def test_config0_tiny(salt_lib, oracle_mod, wl, y_mode):
    w = wl.config0()
    got = run_gpu(w, [[0]], y_mode=y_mode)
    assert_close(got[0], oracle_layer(oracle_mod, w, 0), "config0")


def test_config1_qkv_grouped_and_single(salt_lib, oracle_mod, wl):
    # A grouped launch may split d_in differently from single launches (the
    # split depends on how many (block, projection) pairs share the launch),
    # so the two agree to rounding, each within the tolerance of the oracle.
    w = wl.config1()
    grouped = run_gpu(w, [[0, 1, 2]])
    single = run_gpu(w, [[0], [1], [2]])
    for l in range(3):
        ref = oracle_layer(oracle_mod, w, l)
        assert_close(grouped[l], ref, f"config1 layer {l}, grouped")
        assert_close(single[l], ref, f"config1 layer {l}, single")


def test_config3_layer(salt_lib, oracle_mod, wl):
    w = wl.config3()
    got = run_gpu(w, w.group)
    for l in range(7):
        assert_close(got[l], oracle_layer(oracle_mod, w, l), f"config3 {w.layers[l][0]}")


def test_config2_prefill_sampled_rows(salt_lib, oracle_mod, wl):
    w = wl.config2()
    got = run_gpu(w, w.group)
    ptr = np.flatnonzero(np.r_[True, np.diff(w.slot_ids) != 0])
    rows = np.unique(np.concatenate([ptr, ptr - 1, ptr + 1, ptr + 127, ptr + 128, [0, w.T - 1],
                                     (wl.uniform(2, 555, 96) * w.T).astype(int)]))
    rows = rows[(rows >= 0) & (rows < w.T)]
    for l in range(3):
        assert_close(got[l][rows], oracle_layer(oracle_mod, w, l, rows=rows), f"config2 {w.layers[l][0]}")


def test_prefill_small_full(salt_lib, oracle_mod, wl):
    """Prefill-shaped batch small enough for a full oracle pass: user
    segments of 1..300 tokens, ragged 128-token tiles, rc = 32, r in {1, 2}."""
    lens = [1, 130, 300, 128, 7, 255, 129]
    user = np.repeat(np.arange(len(lens)), lens).astype(np.int32)
    w = wl.Workload("prefill_small", 21, [("gate", 256, 512), ("down", 512, 256)], 4, [32] * 4, len(lens),
                    [1 if u % 2 == 0 else 2 for u in range(len(lens))], dom_ids=user % 4, slot_ids=user,
                    y_mode="normal")
    got = run_gpu(w, [[0], [1]])
    for l in range(2):
        assert_close(got[l], oracle_layer(oracle_mod, w, l), f"prefill_small {l}")


@pytest.mark.parametrize("d_in,d_out", [(8, 8), (72, 40), (520, 1032), (64, 4104)])
def test_ragged_shapes(salt_lib, oracle_mod, wl, d_in, d_out):
    T = 37
    u = (wl.uniform(5, 1, T) * 6).astype(np.int32)
    dom = (u % 3).astype(np.int32)
    dom[::5] = -1
    u[::7] = -1
    w = wl.Workload("ragged", 5, [("p", d_in, d_out)], 3, [8, 24, 64], 6, [1, 2, 2, 1, 2, 2],
                    dom_ids=dom, slot_ids=u, y_mode="normal", s_c=[0.6, 0.8, 1.0], s_u=[1.0, 0.5, 2.0, 1.0, 1.0, 0.25])
    got = run_gpu(w, [[0]])
    assert_close(got[0], oracle_layer(oracle_mod, w, 0), f"ragged {d_in}x{d_out}")


def test_absent_ids_leave_y_bit_identical(salt_lib, oracle_mod, wl):
    T = 40
    dom = np.array([-1, 0, -1, 1] * 10, np.int32)
    slot = np.array([-1, -1, 2, 3] * 10, np.int32)
    w = wl.Workload("absent", 6, [("p", 128, 192)], 2, [16, 16], 4, [2, 2, 1, 2], dom_ids=dom, slot_ids=slot,
                    y_mode="normal")
    y_in = w.y_in(0)
    y_in[0, :8] = 0x8000  # negative zero must survive untouched
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_tensor, bf16_bits
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        x = bf16_tensor(w.x(0))
        y = bf16_tensor(y_in)
        r.apply([0], [x], [y])
        got = bf16_bits(y)
    untouched = (dom == -1) & (slot == -1)
    np.testing.assert_array_equal(got[untouched], y_in[untouched])
    ref = oracle_mod.apply(w.x(0), y_in, dom, slot, *oracle_tables(w, 0))
    assert_close(got, ref, "absent")


def test_rank16_standard_lora(salt_lib, oracle_mod, wl):
    """The comparison mode: no centroid, rank-16 adapters in the slots."""
    T = 96
    k = wl.zipf_draw(wl.uniform(7, 3, T), 24)
    slot = (k - 1).astype(np.int32)
    w = wl.Workload("rank16", 7, [("q", 512, 512), ("k", 512, 128)], 1, [0], 24, [16] * 24,
                    dom_ids=np.full(T, -1, np.int32), slot_ids=slot)
    got = run_gpu(w, [[0, 1]])
    for l in range(2):
        assert_close(got[l], oracle_layer(oracle_mod, w, l), f"rank16 {l}")


def test_centroid_only_and_residual_only(salt_lib, oracle_mod, wl):
    T = 50
    u = (wl.uniform(8, 1, T) * 10).astype(np.int32)
    for dom, slot in [((u % 2).astype(np.int32), np.full(T, -1, np.int32)),
                      (np.full(T, -1, np.int32), u)]:
        w = wl.Workload("split", 8, [("p", 256, 256)], 2, [64, 64], 10, [2] * 10, dom_ids=dom, slot_ids=slot)
        got = run_gpu(w, [[0]])
        assert_close(got[0], oracle_layer(oracle_mod, w, 0), "split")


def test_gamma_bins(salt_lib, oracle_mod, wl):
    w = wl.config0()
    for g in (0.6, 0.8):
        sc = [g, g]
        got = run_gpu(w, [[0]], scales_c=sc)
        assert_close(got[0], oracle_layer(oracle_mod, w, 0, scales_c=sc), f"gamma {g}")


def test_max_tokens_full(salt_lib, oracle_mod, wl):
    T = 16384
    k = wl.zipf_draw(wl.uniform(9, 3, T), 600)
    slot = (k - 1).astype(np.int32)
    w = wl.Workload("maxtok", 9, [("p", 64, 64)], 8, [64] * 8, 600, [2] * 600, dom_ids=slot % 8, slot_ids=slot)
    got = run_gpu(w, [[0]])
    assert_close(got[0], oracle_layer(oracle_mod, w, 0), "max tokens")


def test_deterministic(salt_lib, wl):
    w = wl.config1()
    a = run_gpu(w, [[0, 1, 2]])
    b = run_gpu(w, [[0, 1, 2]])
    for l in range(3):
        np.testing.assert_array_equal(a[l], b[l])


def test_empty_batch_is_noop(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner
    w = wl.Workload("empty", 1, [("p", 64, 64)], 1, [8], 1, [1], dom_ids=np.zeros(0, np.int32),
                    slot_ids=np.zeros(0, np.int32))
    with SaltRunner(w, max_tokens=4) as r:
        r.pin_centroids()
        r.load_slots()
        r.build()
        x = torch.zeros(1, 64, dtype=torch.bfloat16, device="cuda")
        y = torch.ones(1, 64, dtype=torch.bfloat16, device="cuda")
        r.apply([0], [x], [y])
        torch.cuda.synchronize()
        assert (y == 1).all()


def test_apply_argument_errors(salt_lib, wl):
    from paper_2608_03579_gb300.runner import SaltRunner
    salt = salt_lib
    w = wl.config0()
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        seg2 = salt.salt_segments_create(r.ctx)
        x = torch.zeros(16, 512, dtype=torch.bfloat16, device="cuda")
        y = torch.zeros(16, 512, dtype=torch.bfloat16, device="cuda")
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply(r.ctx, seg2, 0, x, y)
        assert e.value.name == "SALT_ERR_NOT_BUILT"
        salt.salt_segments_destroy(seg2)
        r.build()
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply(r.ctx, r.seg, 1, x, y)
        assert e.value.name == "SALT_ERR_LAYER_RANGE"
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply(r.ctx, r.seg, 0, x.data_ptr() + 2, y)
        assert e.value.name == "SALT_ERR_ALIGN"
        with pytest.raises(salt.SaltError) as e:
            salt.salt_lora_apply_grouped(r.ctx, r.seg, [0] * 9, [x] * 9, [y] * 9)
        assert e.value.name == "SALT_ERR_INVALID_ARG"
