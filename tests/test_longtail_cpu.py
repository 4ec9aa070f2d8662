"""The long-tail packer on the host (no GPU): salt_residual_blob_concat
writes the scaled centroid and the residual as one ordinary adapter
(Section "Multi-Tenant Serving": the long-tail form, rank 17 in the paper's
example)."""
import numpy as np
import pytest


def _unpack(blob, din, dout, R):
    hdr = blob[:256]
    pay = blob[256:].view(np.uint16)
    out, off = [], 0
    for a, b in zip(din, dout):
        At = pay[off:off + R * a].reshape(R, a)
        off += R * a
        B = pay[off:off + R * b].reshape(R, b)
        off += R * b
        out.append((At, B))
    return hdr, out


def _factors(wl, seed, rank, din, dout):
    A = wl.normal_bf16(seed, wl.stream_id(96, 1, rank), rank * sum(din), 1 / np.sqrt(din[0]))
    B = wl.normal_bf16(seed, wl.stream_id(96, 2, rank), rank * sum(dout), 1 / np.sqrt(rank))
    return A, B


def _per_layer(flat, rank, dims):
    out, off = [], 0
    for d in dims:
        out.append(flat[off:off + rank * d].reshape(rank, d))
        off += rank * d
    return out


@pytest.mark.parametrize("s_c,s_u", [(1.0, 1.0), (0.8, 2.0), (0.6, 0.0)])
def test_concat_layout_and_scales(salt_lib, wl, s_c, s_u):
    din, dout = [16, 24], [40, 8]
    rc, r = 16, 1
    Ac, Bc = _factors(wl, 1, rc, din, dout)
    Au, Bu = _factors(wl, 2, r, din, dout)
    n = salt_lib.salt_residual_blob_bytes(din, dout, rc + r)
    blob = np.zeros(n, np.uint8)
    salt_lib.salt_residual_blob_concat(din, dout, rc, Ac, Bc, s_c, r, Au, Bu, s_u, blob, n)
    hdr, layers = _unpack(blob, din, dout, rc + r)
    assert hdr[12:16].view(np.int32)[0] == rc + r
    s = s_u if s_u != 0 else 1.0
    assert hdr[20:24].view(np.float32)[0] == np.float32(s)
    Acl, Bcl = _per_layer(Ac, rc, din), _per_layer(Bc, rc, dout)
    Aul, Bul = _per_layer(Au, r, din), _per_layer(Bu, r, dout)
    for l, (At, B) in enumerate(layers):
        np.testing.assert_array_equal(At[:rc], Acl[l])
        np.testing.assert_array_equal(At[rc:], Aul[l])
        fc = np.float32(s_c) / np.float32(s)
        exp_c = Bcl[l] if fc == 1 else wl.float_to_bf16_bits(fc * wl.bf16_bits_to_float(Bcl[l]))
        np.testing.assert_array_equal(B[:rc], exp_c)
        exp_u = Bul[l] if s_u != 0 else np.zeros_like(Bul[l])
        np.testing.assert_array_equal(B[rc:] & (0x7fff if s_u == 0 else 0xffff), exp_u)


def test_concat_is_the_centroid_plus_residual(salt_lib, oracle_mod, wl):
    """Applied as a plain adapter (no centroid), the packed blob gives the
    centroid + residual result up to the one bf16 rounding of the scaled B_c."""
    din, dout = [64], [48]
    rc, r, s_c, s_u = 8, 2, 0.6, 1.0
    Ac, Bc = _factors(wl, 3, rc, din, dout)
    Au, Bu = _factors(wl, 4, r, din, dout)
    n = salt_lib.salt_residual_blob_bytes(din, dout, rc + r)
    blob = np.zeros(n, np.uint8)
    salt_lib.salt_residual_blob_concat(din, dout, rc, Ac, Bc, s_c, r, Au, Bu, s_u, blob, n)
    hdr, [(At, B)] = _unpack(blob, din, dout, rc + r)
    s = float(hdr[20:24].view(np.float32)[0])
    T = 12
    x = wl.normal_bf16(5, wl.stream_id(96, 9), T * din[0]).reshape(T, din[0])
    dom, slot = np.zeros(T, np.int32), np.zeros(T, np.int32)
    ref = oracle_mod.apply(x, None, dom, slot, [(Ac.reshape(rc, -1), Bc.reshape(rc, -1), s_c)],
                           [(Au.reshape(r, -1), Bu.reshape(r, -1), s_u)])
    got = oracle_mod.apply(x, None, np.full(T, -1, np.int32), slot, [None], [(At, B, s)])
    tol = 2e-2 * np.abs(ref) + 2e-2 * np.abs(ref).max()
    assert np.all(np.abs(got - ref) <= tol)
    assert np.abs(got - ref).max() <= 2 ** -8 * np.abs(ref).max()


def test_concat_rejects_ranks_above_the_limit(salt_lib, wl):
    din, dout = [16], [16]
    Ac, Bc = _factors(wl, 6, 64, din, dout)
    Au, Bu = _factors(wl, 7, 17, din, dout)
    n = salt_lib.salt_residual_blob_bytes(din, dout, 81)
    blob = np.zeros(n, np.uint8)
    with pytest.raises(salt_lib.SaltError) as e:
        salt_lib.salt_residual_blob_concat(din, dout, 64, Ac, Bc, 1.0, 17, Au, Bu, 1.0, blob, n)
    assert e.value.name == "SALT_ERR_RANK"
