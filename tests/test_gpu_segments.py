"""Segment builder on the GPU against the grouping oracle: bit-exact."""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

TM = 128


def _ctx(salt, n_domains=9, n_slots=513, max_tokens=16384, r_max=2, rc=16):
    ctx = salt.salt_ctx_create([64], [64], n_domains, rc, n_slots, r_max, max_tokens, 0)
    for d in range(n_domains):
        A = np.zeros(rc * 64, np.uint16)
        salt.salt_centroid_pin(ctx, d, rc, A, A, 1.0)
    blob_n = salt.salt_residual_blob_bytes([64], [64], 1)
    blob = torch.empty(blob_n, dtype=torch.uint8, pin_memory=True)
    z = np.zeros(64, np.uint16)
    salt.salt_residual_blob_pack([64], [64], 1, 1.0, z, z, blob.numpy(), blob_n)
    for s in range(n_slots):
        salt.salt_residual_load(ctx, s, blob, None)
    torch.cuda.synchronize()
    return ctx


@pytest.fixture(scope="module")
def env(salt_lib):
    ctx = _ctx(salt_lib)
    seg = salt_lib.salt_segments_create(ctx)
    yield salt_lib, ctx, seg
    salt_lib.salt_segments_destroy(seg)
    salt_lib.salt_ctx_destroy(ctx)


def _ids(wl, T, nd, ns, seed, p_none=0.15):
    dom = (wl.uniform(seed, wl.stream_id(97, 1), T) * nd).astype(np.int32)
    slot = (wl.uniform(seed, wl.stream_id(97, 2), T) * ns).astype(np.int32)
    dom[wl.uniform(seed, wl.stream_id(97, 3), T) < p_none] = -1
    slot[wl.uniform(seed, wl.stream_id(97, 4), T) < p_none] = -1
    return dom, slot


def _check(salt, ctx, seg, oracle_mod, dom, slot, umax):
    got = salt.salt_segments_export(ctx, seg, 16384)
    ref = oracle_mod.segments(dom, slot)
    for k in ("perm", "dseg_ptr", "dseg_dom", "useg_ptr", "useg_dom", "useg_slot"):
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)
    # row blocks: cover every token except the (-1, -1) run exactly once, in order,
    # each inside one domain run, <= TM tokens and <= umax user runs
    T = len(dom)
    blocks = got["blocks"]
    covered = np.zeros(T, dtype=int)
    useg_ptr = ref["useg_ptr"]
    for (s0, n, d) in blocks:
        assert 1 <= n <= TM
        covered[s0:s0 + n] += 1
        sd = np.asarray(dom)[ref["perm"][s0:s0 + n]]
        assert (sd == d).all()
        runs = np.searchsorted(useg_ptr, np.arange(s0, s0 + n), side="right")
        assert len(np.unique(runs)) <= umax
    skip = np.zeros(T, dtype=bool)
    if T and ref["useg_dom"][0] == -1 and ref["useg_slot"][0] == -1:
        skip[:ref["useg_ptr"][1]] = True
    np.testing.assert_array_equal(covered, (~skip).astype(int))
    if len(blocks) > 1:
        assert (np.diff(blocks[:, 0]) > 0).all()


@pytest.mark.parametrize("T,nd,ns", [(1, 9, 513), (7, 2, 3), (64, 4, 64), (256, 8, 256), (512, 8, 448),
                                     (1000, 3, 20), (4096, 9, 513), (8192, 4, 14), (16384, 9, 513)])
def test_segments_host_ids(env, oracle_mod, wl, T, nd, ns):
    salt, ctx, seg = env
    dom, slot = _ids(wl, T, nd, ns, seed=T)
    salt.salt_build_segments(ctx, seg, dom, slot)
    _check(salt, ctx, seg, oracle_mod, dom, slot, umax=(128 - 16) // 2)
    assert salt.salt_get_device_error(ctx) == 0


@pytest.mark.parametrize("T", [33, 700, 16384])
def test_segments_device_ids(env, oracle_mod, wl, T):
    salt, ctx, seg = env
    dom, slot = _ids(wl, T, 9, 513, seed=T + 1)
    dd = torch.from_numpy(dom).cuda()
    ds = torch.from_numpy(slot).cuda()
    salt.salt_build_segments(ctx, seg, dd, ds)
    _check(salt, ctx, seg, oracle_mod, dom, slot, umax=(128 - 16) // 2)
    assert salt.salt_get_device_error(ctx) == 0


def test_segments_degenerate(env, oracle_mod):
    salt, ctx, seg = env
    for dom, slot in [(np.zeros(0, np.int32), np.zeros(0, np.int32)),
                      (np.full(50, -1, np.int32), np.full(50, -1, np.int32)),
                      (np.full(300, 3, np.int32), np.full(300, 7, np.int32)),
                      (np.full(129, -1, np.int32), np.arange(129, dtype=np.int32)),
                      (np.arange(8, dtype=np.int32)[::-1].copy(), np.full(8, -1, np.int32))]:
        salt.salt_build_segments(ctx, seg, dom, slot)
        _check(salt, ctx, seg, oracle_mod, dom, slot, umax=(128 - 16) // 2)


def test_host_id_errors(env):
    salt, ctx, seg = env
    ok = np.zeros(4, np.int32)
    for dom, slot, name in [(np.array([0, 9, 0, 0], np.int32), ok, "SALT_ERR_DOMAIN_RANGE"),
                            (ok, np.array([0, 0, 513, 0], np.int32), "SALT_ERR_SLOT_RANGE"),
                            (ok, np.array([0, -2, 0, 0], np.int32), "SALT_ERR_SLOT_RANGE")]:
        with pytest.raises(salt.SaltError) as e:
            salt.salt_build_segments(ctx, seg, dom, slot)
        assert e.value.name == name
    with pytest.raises(salt.SaltError) as e:
        salt.salt_build_segments(ctx, seg, np.zeros(16385, np.int32), np.zeros(16385, np.int32))
    assert e.value.name == "SALT_ERR_TOO_MANY_TOKENS"


def test_device_id_errors_raise_flags(salt_lib, oracle_mod):
    salt = salt_lib
    ctx = salt.salt_ctx_create([64], [64], 4, 8, 8, 2, 64, 0)
    try:
        A = np.zeros(8 * 64, np.uint16)
        salt.salt_centroid_pin(ctx, 0, 8, A, A, 1.0)  # domains 1..3 stay unpinned; no slot is loaded
        seg = salt.salt_segments_create(ctx)
        dom = torch.tensor([0, 7, 1, 0, -1], dtype=torch.int32, device="cuda")
        slot = torch.tensor([-1, -1, -1, 3, 9], dtype=torch.int32, device="cuda")
        salt.salt_build_segments(ctx, seg, dom, slot)
        flags = salt.salt_get_device_error(ctx)
        assert flags & 0x1  # domain 7 out of range
        assert flags & 0x2  # domain 1 not pinned
        assert flags & 0x4  # slot 9 out of range
        assert flags & 0x8  # slot 3 never loaded
        assert salt.salt_get_device_error(ctx) == 0  # cleared
        # invalid ids were treated as -1: the grouping equals the oracle's on the sanitised ids
        got = salt.salt_segments_export(ctx, seg, 64)
        ref = oracle_mod.segments(np.array([0, -1, -1, 0, -1], np.int32), np.array([-1, -1, -1, -1, -1], np.int32))
        np.testing.assert_array_equal(got["perm"], ref["perm"])
        salt.salt_segments_destroy(seg)
        # the host path reports the same problems at once
        seg = salt.salt_segments_create(ctx)
        with pytest.raises(salt.SaltError) as e:
            salt.salt_build_segments(ctx, seg, np.array([1], np.int32), np.array([-1], np.int32))
        assert e.value.name == "SALT_ERR_DOMAIN_NOT_PINNED"
        with pytest.raises(salt.SaltError) as e:
            salt.salt_build_segments(ctx, seg, np.array([0], np.int32), np.array([3], np.int32))
        assert e.value.name == "SALT_ERR_SLOT_EMPTY"
        salt.salt_segments_destroy(seg)
    finally:
        salt.salt_ctx_destroy(ctx)
