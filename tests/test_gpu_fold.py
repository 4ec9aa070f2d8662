"""Centroid fold on the GPU (Section "Multi-Tenant Serving": a scaled
centroid fused into the base weight) against the fp64 oracle."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


def _setup(salt, wl, din, dout, rc, s_c, seed):
    ctx = salt.salt_ctx_create([din], [dout], 2, rc, 1, 1, 16, 0)
    A = wl.normal_bf16(seed, wl.stream_id(94, 1), rc * din, 1 / np.sqrt(din))
    B = wl.normal_bf16(seed, wl.stream_id(94, 2), rc * dout, 1 / np.sqrt(rc))
    salt.salt_centroid_pin(ctx, 1, rc, A, B, s_c)
    return ctx, A.reshape(rc, din), B.reshape(rc, dout)


def _ulp_check(got_bits, ref, w0_bits, wl):
    """One rounding to bf16: within one unit in the last place of the
    reference, plus the fp32 arithmetic before it (relative 2^-20 of the
    operands |W| + |delta|, a generous bound on the fp32 accumulation)."""
    g = wl.bf16_bits_to_float(got_bits).astype(np.float64)
    w0 = wl.bf16_bits_to_float(w0_bits).astype(np.float64)
    slack = np.abs(ref) * 2.0 ** -7 + (np.abs(w0) + np.abs(ref - w0)) * 2.0 ** -20
    assert (np.abs(g - ref) <= slack).all(), np.abs(g - ref).max()


@pytest.mark.parametrize("layout", [0, 1])
@pytest.mark.parametrize("din,dout,rc", [(328, 200, 13), (128, 64, 64), (8, 8, 1), (1032, 520, 48)])
def test_fold_matches_oracle(salt_lib, oracle_mod, wl, layout, din, dout, rc):
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    ctx, A, B = _setup(salt, wl, din, dout, rc, 0.75, seed=din + rc)
    try:
        shape = (din, dout) if layout == 0 else (dout, din)
        W0 = wl.normal_bf16(3, wl.stream_id(94, 3, layout), din * dout).reshape(shape)
        W = bf16_tensor(W0)
        salt.salt_centroid_fold(ctx, 1, 0, 0.8, W, layout)
        torch.cuda.synchronize()
        ref = oracle_mod.fold(A, B, float(np.float32(0.8) * np.float32(0.75)), W0, layout)
        got = bf16_bits(W)
        assert_close(got, ref, "fold")
        _ulp_check(got, ref, W0, wl)
        assert salt.salt_get_device_error(ctx) == 0
    finally:
        salt.salt_ctx_destroy(ctx)


def test_fold_then_unfold(salt_lib, wl):
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    ctx, A, B = _setup(salt, wl, 512, 384, 32, 1.0, seed=5)
    try:
        W0 = wl.normal_bf16(5, wl.stream_id(94, 4), 512 * 384).reshape(512, 384)
        W = bf16_tensor(W0)
        salt.salt_centroid_fold(ctx, 1, 0, 0.6, W, 0)
        assert not np.array_equal(bf16_bits(W), W0)
        salt.salt_centroid_fold(ctx, 1, 0, -0.6, W, 0)
        torch.cuda.synchronize()
        g = wl.bf16_bits_to_float(bf16_bits(W)).astype(np.float64)
        w0 = wl.bf16_bits_to_float(W0).astype(np.float64)
        delta = np.abs(0.6 * (wl.bf16_bits_to_float(A).astype(np.float64).T @ wl.bf16_bits_to_float(B)))
        # two roundings, each at most half a unit of a value below |W| + |delta|
        assert (np.abs(g - w0) <= (np.abs(w0) + delta) * 2.0 ** -7 + 1e-30).all()
    finally:
        salt.salt_ctx_destroy(ctx)


@pytest.mark.parametrize("name,din,dout,layout", [("gate", 4096, 14336, 0), ("down", 14336, 4096, 1)])
def test_fold_llama8b_full_size(salt_lib, oracle_mod, wl, name, din, dout, layout):
    """A full Llama-3.1-8B projection with the rank-64 centroid; sampled rows
    of W (in its own layout) against the oracle."""
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    ctx, A, B = _setup(salt, wl, din, dout, 64, 1.0, seed=11)
    try:
        shape = (din, dout) if layout == 0 else (dout, din)
        W0 = wl.normal_bf16(11, wl.stream_id(94, 5, layout), din * dout).reshape(shape)
        W = bf16_tensor(W0)
        salt.salt_centroid_fold(ctx, 1, 0, 0.8, W, layout)
        torch.cuda.synchronize()
        got = bf16_bits(W)
        rows = np.unique(np.r_[0, 1, 127, 128, shape[0] - 1, (wl.uniform(11, wl.stream_id(94, 6), 12) * shape[0]).astype(int)])
        if layout == 0:
            ref = oracle_mod.fold(np.ascontiguousarray(A[:, rows]), B, 0.8, W0[rows], 0)
        else:
            ref = oracle_mod.fold(A, np.ascontiguousarray(B[:, rows]), 0.8, W0[rows], 1)
        assert_close(got[rows], ref, f"{name} fold")
        _ulp_check(got[rows], ref, W0[rows], wl)
        assert salt.salt_get_device_error(ctx) == 0
    finally:
        salt.salt_ctx_destroy(ctx)


def test_fold_argument_errors(salt_lib, wl):
    from paper_2608_03579_gb300.runner import bf16_tensor
    salt = salt_lib
    ctx, A, B = _setup(salt, wl, 64, 64, 8, 1.0, seed=2)
    try:
        W = bf16_tensor(np.zeros((64, 64), np.uint16))
        for args, name in [((0, 0, 1.0, W, 0), "SALT_ERR_DOMAIN_NOT_PINNED"),
                           ((2, 0, 1.0, W, 0), "SALT_ERR_DOMAIN_RANGE"),
                           ((1, 1, 1.0, W, 0), "SALT_ERR_LAYER_RANGE"),
                           ((1, 0, 1.0, W, 2), "SALT_ERR_INVALID_ARG"),
                           ((1, 0, 1.0, W.data_ptr() + 2, 0), "SALT_ERR_ALIGN")]:
            with pytest.raises(salt.SaltError) as e:
                salt.salt_centroid_fold(ctx, *args)
            assert e.value.name == name
    finally:
        salt.salt_ctx_destroy(ctx)


def _plan_setup(salt, wl, shapes, rc, s_c, seed):
    ctx = salt.salt_ctx_create([a for a, _ in shapes], [b for _, b in shapes], 2, 64, 1, 1, 16, 0)
    As = [wl.normal_bf16(seed, wl.stream_id(95, 1, l), rc * a, 1 / np.sqrt(a)) for l, (a, _) in enumerate(shapes)]
    Bs = [wl.normal_bf16(seed, wl.stream_id(95, 2, l), rc * b, 1 / np.sqrt(rc)) for l, (_, b) in enumerate(shapes)]
    salt.salt_centroid_pin(ctx, 1, rc, np.concatenate(As), np.concatenate(Bs), s_c)
    return ctx, [A.reshape(rc, a) for A, (a, _) in zip(As, shapes)], [B.reshape(rc, b) for B, (_, b) in zip(Bs, shapes)]


@pytest.mark.parametrize("layout", [0, 1])
def test_fold_plan_equals_single_folds(salt_lib, oracle_mod, wl, layout):
    """One plan launch over weights of five ragged shapes (one layer twice,
    with two weights) is bit-identical to a salt_centroid_fold per weight,
    for +gamma and then -gamma; two weights also against the oracle."""
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    shapes = [(328, 200), (128, 64), (1032, 520), (8, 8), (4096, 1024)]
    layers = [0, 1, 2, 3, 4, 2]
    ctx, As, Bs = _plan_setup(salt, wl, shapes, 40, 0.75, seed=21)
    plan = None
    try:
        W0 = []
        for i, l in enumerate(layers):
            a, b = shapes[l]
            W0.append(wl.normal_bf16(21, wl.stream_id(95, 3, i, layout), a * b).reshape((a, b) if layout == 0 else (b, a)))
        Wp = [bf16_tensor(w) for w in W0]
        Ws = [bf16_tensor(w) for w in W0]
        plan = salt.salt_fold_plan_create(ctx, 1, layers, Wp, layout)
        for g in (0.8, -0.8):
            salt.salt_fold_plan_run(plan, g)
            for i, l in enumerate(layers):
                salt.salt_centroid_fold(ctx, 1, l, g, Ws[i], layout)
            torch.cuda.synchronize()
            for i in range(len(layers)):
                assert np.array_equal(bf16_bits(Wp[i]), bf16_bits(Ws[i])), (g, i)
            if g > 0:
                for i in (0, 4):
                    l = layers[i]
                    ref = oracle_mod.fold(As[l], Bs[l], float(np.float32(0.8) * np.float32(0.75)), W0[i], layout)
                    assert_close(bf16_bits(Wp[i]), ref, f"plan fold weight {i}")
                    _ulp_check(bf16_bits(Wp[i]), ref, W0[i], wl)
        assert salt.salt_get_device_error(ctx) == 0
    finally:
        salt.salt_fold_plan_destroy(plan)
        salt.salt_ctx_destroy(ctx)


def test_fold_plan_errors(salt_lib, wl):
    from paper_2608_03579_gb300.runner import bf16_tensor
    salt = salt_lib
    shapes = [(64, 64), (128, 64)]
    ctx, As, Bs = _plan_setup(salt, wl, shapes, 8, 1.0, seed=3)
    try:
        W = bf16_tensor(np.zeros((64, 64), np.uint16))
        W2 = bf16_tensor(np.zeros((128, 64), np.uint16))
        big = bf16_tensor(np.zeros((256, 64), np.uint16))
        for args, name in [((1, [0, 0], [W, W], 0), "SALT_ERR_INVALID_ARG"),          # the same weight twice
                           ((1, [0, 1], [big[64:128], big[96:224]], 0), "SALT_ERR_INVALID_ARG"),  # overlap
                           ((1, [0, 2], [W, W2], 0), "SALT_ERR_LAYER_RANGE"),
                           ((0, [0], [W], 0), "SALT_ERR_DOMAIN_NOT_PINNED"),
                           ((1, [0], [W], 3), "SALT_ERR_INVALID_ARG"),
                           ((1, [], [], 0), "SALT_ERR_INVALID_ARG")]:
            with pytest.raises(salt.SaltError) as e:
                salt.salt_fold_plan_create(ctx, *args)
            assert e.value.name == name, (args, e.value.name)
        plan = salt.salt_fold_plan_create(ctx, 1, [0, 1], [W, W2], 0)
        try:
            salt.salt_fold_plan_run(plan, 0.5)
            # re-pinned with another rank: the plan refuses to run
            rc2 = 16
            salt.salt_centroid_pin(ctx, 1, rc2,
                                   np.concatenate([wl.normal_bf16(4, wl.stream_id(95, 9, l), rc2 * a, 0.1) for l, (a, _) in enumerate(shapes)]),
                                   np.concatenate([wl.normal_bf16(4, wl.stream_id(95, 10, l), rc2 * b, 0.1) for l, (_, b) in enumerate(shapes)]),
                                   1.0)
            with pytest.raises(salt.SaltError) as e:
                salt.salt_fold_plan_run(plan, 0.5)
            assert e.value.name == "SALT_ERR_RANK"
        finally:
            salt.salt_fold_plan_destroy(plan)
        torch.cuda.synchronize()
        assert salt.salt_get_device_error(ctx) == 0
    finally:
        salt.salt_ctx_destroy(ctx)
