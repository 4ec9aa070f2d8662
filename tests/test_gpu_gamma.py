"""Gamma bins on the GPU (Section "Multi-Tenant Serving": requests are
grouped by their (centroid, gamma) pair, gamma from a small fixed set of bins).
The grouping is compared bit for bit with the oracle; the apply with
per-token gamma within the serving tolerance."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close, oracle_tables

pytestmark = pytest.mark.gpu

TM = 128


@pytest.fixture(scope="module")
def env(salt_lib):
    salt = salt_lib
    n_domains, n_slots, rc = 9, 513, 16
    ctx = salt.salt_ctx_create([64], [64], n_domains, rc, n_slots, 2, 16384, 0)
    A = np.zeros(rc * 64, np.uint16)
    for d in range(n_domains):
        salt.salt_centroid_pin(ctx, d, rc, A, A, 1.0)
    blob_n = salt.salt_residual_blob_bytes([64], [64], 1)
    blob = torch.empty(blob_n, dtype=torch.uint8, pin_memory=True)
    z = np.zeros(64, np.uint16)
    salt.salt_residual_blob_pack([64], [64], 1, 1.0, z, z, blob.numpy(), blob_n)
    for s in range(n_slots):
        salt.salt_residual_load(ctx, s, blob, None)
    torch.cuda.synchronize()
    seg = salt.salt_segments_create(ctx)
    yield salt, ctx, seg
    salt.salt_segments_destroy(seg)
    salt.salt_ctx_destroy(ctx)


def _ids(wl, T, nd, ns, nb, seed):
    dom = (wl.uniform(seed, wl.stream_id(95, 1), T) * (nd + 1)).astype(np.int32) - 1
    slot = (wl.uniform(seed, wl.stream_id(95, 2), T) * (ns + 1)).astype(np.int32) - 1
    gb = (wl.uniform(seed, wl.stream_id(95, 3), T) * (nb + 1)).astype(np.int32) - 1
    return dom, slot, gb


def _check(salt, ctx, seg, oracle_mod, dom, slot, gb):
    got = salt.salt_segments_export(ctx, seg, 16384)
    got.update(salt.salt_segments_export_gamma(ctx, seg, 16384))
    ref = oracle_mod.segments(dom, slot, gb)
    for k in ("perm", "dseg_ptr", "dseg_dom", "dseg_gbin", "useg_ptr", "useg_dom", "useg_gbin", "useg_slot"):
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)
    # row blocks: inside one domain (a block may span the domain's bins: gamma
    # is applied per token), consecutive, covering every token with a term once
    covered = np.zeros(len(dom), dtype=int)
    for (s0, n, d) in got["blocks"]:
        assert 1 <= n <= TM
        toks = ref["perm"][s0:s0 + n]
        assert (dom[toks] == d).all()
        covered[s0:s0 + n] += 1
    active = (dom[ref["perm"]] >= 0) | (slot[ref["perm"]] >= 0)
    np.testing.assert_array_equal(covered, active.astype(int))
    # The blocks index the apply order: the same tokens stably sorted by
    # (domain, slot, bin), so that a user's tokens in several bins are one
    # run of its block and a block holds at most umax distinct users (here
    # (128 - 16) / 2 = 56), however many bins they span.
    dom, slot, gb = (np.asarray(a) for a in (dom, slot, gb))
    gbk = np.where(dom >= 0, gb, -1)
    apply_order = np.lexsort((np.arange(len(dom)), gbk, slot, dom))
    for (s0, n, d) in got["blocks"]:
        toks = apply_order[s0:s0 + n]
        assert (dom[toks] == d).all()
        sl = slot[toks]
        users = np.unique(sl[sl >= 0])
        assert len(users) <= (TM - 16) // 2
        runs = 1 + int(np.count_nonzero(np.diff(sl)))  # every user's tokens are contiguous
        assert runs == len(np.unique(sl))


@pytest.mark.parametrize("T", [1, 77, 512, 4096, 16384])
def test_gamma_segments_host_ids(env, oracle_mod, wl, T):
    salt, ctx, seg = env
    dom, slot, gb = _ids(wl, T, 9, 513, 3, seed=T)
    salt.salt_build_segments_gamma(ctx, seg, dom, gb, slot, wl.GAMMA_BINS)
    _check(salt, ctx, seg, oracle_mod, dom, slot, gb)
    assert salt.salt_get_device_error(ctx) == 0


@pytest.mark.parametrize("T", [300, 16384])
def test_gamma_segments_device_ids(env, oracle_mod, wl, T):
    salt, ctx, seg = env
    dom, slot, gb = _ids(wl, T, 9, 513, 16, seed=T + 7)
    gammas = [0.1 * (i + 1) for i in range(16)]
    salt.salt_build_segments_gamma(ctx, seg, torch.from_numpy(dom).cuda(), torch.from_numpy(gb).cuda(),
                                   torch.from_numpy(slot).cuda(), gammas)
    _check(salt, ctx, seg, oracle_mod, dom, slot, gb)
    assert salt.salt_get_device_error(ctx) == 0


def test_gamma_bin_range(env, oracle_mod):
    salt, ctx, seg = env
    dom = np.array([0, 1, -1, 2], np.int32)
    slot = np.array([0, -1, 3, 4], np.int32)
    bad = np.array([0, 3, 7, -1], np.int32)  # bin 3 of token 1 is outside [-1, 3); token 2 has no centroid
    with pytest.raises(salt.SaltError) as e:
        salt.salt_build_segments_gamma(ctx, seg, dom, bad, slot, [0.6, 0.8, 1.0])
    assert e.value.name == "SALT_ERR_GAMMA_RANGE"
    # on the device the bin is flagged and taken as -1
    salt.salt_build_segments_gamma(ctx, seg, torch.from_numpy(dom).cuda(), torch.from_numpy(bad).cuda(),
                                   torch.from_numpy(slot).cuda(), [0.6, 0.8, 1.0])
    assert salt.salt_get_device_error(ctx) & 0x40
    fixed = np.array([0, -1, 7, -1], np.int32)
    _check(salt, ctx, seg, oracle_mod, dom, slot, fixed)
    # a centroid-less token's bin is never checked
    salt.salt_build_segments_gamma(ctx, seg, dom, np.array([0, 2, 99, 1], np.int32), slot, [0.6, 0.8, 1.0])
    assert salt.salt_get_device_error(ctx) == 0


@pytest.mark.parametrize("static", [False, True])
def test_gamma_apply_llama8b_layer(salt_lib, oracle_mod, wl, static):
    """Llama-3.1-8B layer, 256 decode tokens, each with a bin of
    {0.6, 0.8, 1.0} or none: y += gamma s_c (x A_c) B_c + s_u (x a_u) b_u."""
    from paper_2608_03579_gb300.runner import SaltRunner, bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config3()
    w.y_mode = "normal"
    gb = wl.gamma_bin_ids(w.seed, w.T, 3, p_none=0.2)
    gamma_t = np.where(gb >= 0, np.array(wl.GAMMA_BINS)[np.maximum(gb, 0)], 1.0)
    layers = [0, 3, 4] if static else list(range(7))
    with SaltRunner(w) as r:
        r.pin_centroids()
        r.load_slots()
        salt.salt_build_segments_gamma(r.ctx, r.seg, w.dom_ids, gb, w.slot_ids, wl.GAMMA_BINS)
        for grp in ([[l] for l in layers] if static else w.group):
            xs, ys = r.alloc_xy(grp)
            if static:
                salt.salt_lora_apply_static(r.ctx, r.seg, grp[0], xs[0], ys[0])
            else:
                r.apply(grp, xs, ys)
            torch.cuda.synchronize()
            for l, y in zip(grp, ys):
                cents, res = oracle_tables(w, l)
                ref = oracle_mod.apply(w.x(l), w.y_in(l), w.dom_ids, w.slot_ids, cents, res, gamma=gamma_t)
                assert_close(bf16_bits(y), ref, f"gamma apply, projection {l}")
        assert r.device_error() == 0
