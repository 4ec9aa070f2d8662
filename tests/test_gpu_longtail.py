"""Long-tail requests on the GPU (Section "Multi-Tenant Serving": the scaled
centroid and the residual stacked ahead of time into one ordinary adapter,
served like any other adapter of a mixed batch) and residual ranks above 16."""
import numpy as np
import pytest
import torch

from gpu_helpers import assert_close

pytestmark = pytest.mark.gpu


def _cat_blobs(salt, wl, w, pairs, s_c, s_u):
    """One concatenated blob per (domain, slot) pair, in page-locked memory."""
    blobs = []
    for (d, u) in pairs:
        Ac, Bc = w.centroid_packed(d)
        Au, Bu = w.residual_packed(u)
        R = w.rc[d] + w.r_u[u]
        n = salt.salt_residual_blob_bytes(w.d_in, w.d_out, R)
        blob = torch.empty(n, dtype=torch.uint8, pin_memory=True)
        salt.salt_residual_blob_concat(w.d_in, w.d_out, w.rc[d], Ac, Bc, s_c, w.r_u[u], Au, Bu, s_u, blob.numpy(), n)
        blobs.append(blob)
    return blobs


def _oracle(oracle_mod, w, l, T, s_c, s_u):
    """The first T tokens of the workload as centroid + residual."""
    cents = [(w.centroid_At(d, l), w.centroid_B(d, l), s_c) for d in range(w.n_domains)]
    res = [(w.residual_At(u, l), w.residual_B(u, l), s_u) for u in range(w.n_slots)]
    return oracle_mod.apply(w.x(l)[:T], None, w.dom_ids[:T], w.slot_ids[:T], cents, res)


@pytest.mark.parametrize("s_c", [0.8, 1.0])
def test_rank66_concatenation_llama8b_layer(salt_lib, oracle_mod, wl, s_c):
    """Rank-64 centroid + rank-2 residual of the Llama-3.1-8B layer as one
    rank-66 adapter per (domain, user), applied with no centroid, equals the
    centroid + residual result."""
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    w = wl.config3()
    T = 96
    pairs = sorted(set(zip(w.dom_ids[:T].tolist(), w.slot_ids[:T].tolist())))
    blobs = _cat_blobs(salt, wl, w, pairs, s_c, 1.0)
    idx = {p: i for i, p in enumerate(pairs)}
    cat_slot = np.array([idx[(d, u)] for d, u in zip(w.dom_ids[:T], w.slot_ids[:T])], np.int32)
    ctx = salt.salt_ctx_create(w.d_in, w.d_out, 1, 0, len(pairs), 66, T, 0)
    try:
        seg = salt.salt_segments_create(ctx)
        for i, b in enumerate(blobs):
            salt.salt_residual_load(ctx, i, b, None)
        torch.cuda.synchronize()
        salt.salt_build_segments(ctx, seg, np.full(T, -1, np.int32), cat_slot)
        for l in range(7):
            x = bf16_tensor(w.x(l)[:T])
            y = bf16_tensor(np.zeros((T, w.d_out[l]), np.uint16))
            salt.salt_lora_apply(ctx, seg, l, x, y)
            torch.cuda.synchronize()
            ref = _oracle(oracle_mod, w, l, T, s_c, 1.0)
            assert_close(bf16_bits(y), ref, f"rank-66 concatenation, projection {l}")
        assert salt.salt_get_device_error(ctx) == 0
        salt.salt_segments_destroy(seg)
    finally:
        salt.salt_ctx_destroy(ctx)


def test_mixed_pinned_and_long_tail_batch(salt_lib, oracle_mod, wl):
    """One batch, one context (rc_max 16, r_max 64): requests of pinned
    rank-16 centroids with rank-2 residuals next to long-tail requests that
    carry their rank-17 concatenation (16 + 1) and rank-40 plain adapters."""
    from paper_2608_03579_gb300.runner import bf16_bits, bf16_tensor
    salt = salt_lib
    d_in, d_out = [3072, 3072], [1024, 8192]
    T, n_dom = 200, 3
    sid = wl.stream_id

    def fac(kind, i, r, l):
        di, do = d_in[l], d_out[l]
        A = wl.normal_bf16(8, sid(92, kind, i, l), r * di, 1 / np.sqrt(di)).reshape(r, di)
        B = wl.normal_bf16(8, sid(92, kind + 1, i, l), r * do, 1 / np.sqrt(r)).reshape(r, do)
        return A, B

    cent = [[fac(1, d, 16, l) for l in range(2)] for d in range(n_dom)]
    small = [[fac(3, u, 2, l) for l in range(2)] for u in range(6)]   # rank-2 residuals, slots 0..5
    tail_res = [[fac(5, u, 1, l) for l in range(2)] for u in range(3)]  # rank-1 residuals of the long tail
    plain = [[fac(7, u, 40, l) for l in range(2)] for u in range(2)]    # rank-40 standard adapters
    ctx = salt.salt_ctx_create(d_in, d_out, n_dom, 16, 11, 64, T, 0)
    try:
        packed = lambda fs, k: np.concatenate([f[k].ravel() for f in fs])
        for d in range(n_dom):
            salt.salt_centroid_pin(ctx, d, 16, packed(cent[d], 0), packed(cent[d], 1), 0.8)
        blobs = []
        for u in range(6):
            n = salt.salt_residual_blob_bytes(d_in, d_out, 2)
            b = torch.empty(n, dtype=torch.uint8, pin_memory=True)
            salt.salt_residual_blob_pack(d_in, d_out, 2, 1.0, packed(small[u], 0), packed(small[u], 1), b.numpy(), n)
            blobs.append(b)
        for u in range(3):  # slots 6..8: centroid (u % 3) concatenated with tail residual u
            n = salt.salt_residual_blob_bytes(d_in, d_out, 17)
            b = torch.empty(n, dtype=torch.uint8, pin_memory=True)
            salt.salt_residual_blob_concat(d_in, d_out, 16, packed(cent[u], 0), packed(cent[u], 1), 0.8, 1,
                                           packed(tail_res[u], 0), packed(tail_res[u], 1), 1.0, b.numpy(), n)
            blobs.append(b)
        for u in range(2):  # slots 9..10
            n = salt.salt_residual_blob_bytes(d_in, d_out, 40)
            b = torch.empty(n, dtype=torch.uint8, pin_memory=True)
            salt.salt_residual_blob_pack(d_in, d_out, 40, 0.5, packed(plain[u], 0), packed(plain[u], 1), b.numpy(), n)
            blobs.append(b)
        for s, b in enumerate(blobs):
            salt.salt_residual_load(ctx, s, b, None)
        torch.cuda.synchronize()
        kind = (wl.uniform(8, sid(92, 20), T) * 3).astype(int)
        pick = (wl.uniform(8, sid(92, 21), T) * 6).astype(int)
        dom = np.where(kind == 0, pick % n_dom, -1).astype(np.int32)
        slot = np.where(kind == 0, pick, np.where(kind == 1, 6 + pick % 3, 9 + pick % 2)).astype(np.int32)
        seg = salt.salt_segments_create(ctx)
        salt.salt_build_segments(ctx, seg, dom, slot)
        for l in range(2):
            x_bits = wl.normal_bf16(8, sid(92, 30, l), T * d_in[l]).reshape(T, d_in[l])
            y = bf16_tensor(np.zeros((T, d_out[l]), np.uint16))
            salt.salt_lora_apply(ctx, seg, l, bf16_tensor(x_bits), y)
            torch.cuda.synchronize()
            # oracle: the long-tail tokens as the centroid + residual they stand for
            o_dom = np.where(kind == 1, slot - 6, dom).astype(np.int32)
            o_slot = slot  # slots 6..8 stand for their rank-1 tail residuals
            cents = [(cent[d][l][0], cent[d][l][1], 0.8) for d in range(n_dom)]
            res = ([(small[u][l][0], small[u][l][1], 1.0) for u in range(6)] +
                   [(tail_res[u][l][0], tail_res[u][l][1], 1.0) for u in range(3)] +
                   [(plain[u][l][0], plain[u][l][1], 0.5) for u in range(2)])
            ref = oracle_mod.apply(x_bits, None, o_dom, o_slot, cents, res)
            assert_close(bf16_bits(y), ref, f"mixed batch, layer {l}")
        assert salt.salt_get_device_error(ctx) == 0
        salt.salt_segments_destroy(seg)
    finally:
        salt.salt_ctx_destroy(ctx)
