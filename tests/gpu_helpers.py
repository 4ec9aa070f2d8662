"""Shared helpers of the GPU parity tests: oracle tables and the tolerance.

Tolerance of the serving path (bf16 inputs with fp32 accumulation):
|y_gpu - y_ref| <= 2e-2 * |y_ref| + 2e-2 * max|y_ref|, the max taken over the
output tensor of the call (or of the sampled rows).  Index outputs are
compared bit for bit.
"""
import numpy as np

from paper_2608_03579_gb300.workloads import bf16_bits_to_float

RTOL = 2e-2
ATOL_OF_MAX = 2e-2


def oracle_tables(wl, l, version=0, slots=None, scales_c=None, scales_u=None, rank_override=None):
    cents = []
    for d in range(wl.n_domains):
        if wl.rc[d] <= 0:
            cents.append(None)
            continue
        s = wl.s_c[d] if scales_c is None else scales_c[d]
        cents.append((wl.centroid_At(d, l), wl.centroid_B(d, l), s))
    res = []
    for u in range(wl.n_slots):
        r = wl.r_u[u] if rank_override is None else rank_override
        if r <= 0 or (slots is not None and u not in slots):
            res.append(None)
            continue
        v = version(u) if callable(version) else version
        s = wl.s_u[u] if scales_u is None else scales_u[u]
        res.append((wl.residual_At(u, l, v, r), wl.residual_B(u, l, v, r), s))
    return cents, res


def assert_close(y_bits, y_ref, what=""):
    g = bf16_bits_to_float(np.asarray(y_bits)).astype(np.float64)
    ref = np.asarray(y_ref, dtype=np.float64)
    assert g.shape == ref.shape, (g.shape, ref.shape)
    if ref.size == 0:
        return
    tol = RTOL * np.abs(ref) + ATOL_OF_MAX * np.abs(ref).max()
    err = np.abs(g - ref)
    bad = err > tol
    assert not bad.any(), (f"{what}: {bad.sum()} of {bad.size} elements out of tolerance; "
                           f"worst err {err.max():.4g} (ref max {np.abs(ref).max():.4g}) at {np.unravel_index(err.argmax(), err.shape)}")
    return float((err / (np.abs(ref).max() + 1e-30)).max())


GUARD_ELEMS = 2048          # 4 KiB of bf16 on each side of a guarded buffer
GUARD_BITS = 0x5AA5


def guarded_like(t):
    """A copy of the device tensor t inside a larger buffer whose 4 KiB on
    each side hold a fixed pattern; returns (view of the copy, buffer)."""
    import torch
    n = t.numel()
    buf = torch.empty(n + 2 * GUARD_ELEMS, dtype=t.dtype, device=t.device)
    buf.view(torch.int16).fill_(GUARD_BITS - (1 << 16) if GUARD_BITS >= (1 << 15) else GUARD_BITS)
    view = buf[GUARD_ELEMS:GUARD_ELEMS + n].view(t.shape)
    view.copy_(t)
    return view, buf


def guards_intact(buf) -> bool:
    """True when both bands of a guarded_like buffer still hold the pattern."""
    import torch
    b = buf.view(torch.int16)
    pat = GUARD_BITS - (1 << 16) if GUARD_BITS >= (1 << 15) else GUARD_BITS
    return bool((b[:GUARD_ELEMS] == pat).all().item() and (b[-GUARD_ELEMS:] == pat).all().item())
