"""fp64 CPU oracle for the SALT serving path (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
product library never loads it, and it imports nothing from the product
package: the two share no code.  The arithmetic lives in ``salt_oracle.c``
(plain C, double precision); this module only compiles it with the host C
compiler and marshals numpy arrays through ctypes.

Paper sections followed: "Multi-Tenant Serving" (W_final = W_base +
gamma*Wbar + delta_i, the grouping of requests by their (centroid, gamma)
pair, the fold of a scaled centroid into the base weights), "The
Centroid-Residual Decomposition" (Wbar and delta_i as low-rank products),
Eq. 2 (the alignment regulariser of Phase 1) and the memory columns of
Table 1 and the appendix tables (adapter bytes).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "salt_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libsalt_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``salt_oracle.c`` into ``libsalt_oracle.so`` next to it."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
           "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _configure(lib):
    vp = ctypes.c_void_p
    i32, i64 = ctypes.c_int32, ctypes.c_int64
    lib.oracle_apply.restype = ctypes.c_int
    lib.oracle_apply.argtypes = [i64, i64, i64, vp, vp, vp, i32, vp, vp, vp,
                                 i32, vp, vp, vp, vp,
                                 i32, vp, vp, vp, vp,
                                 i64, vp, vp]
    lib.oracle_segments.restype = ctypes.c_int
    lib.oracle_segments.argtypes = [i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    f64 = ctypes.c_double
    lib.oracle_align_loss.restype = ctypes.c_int
    lib.oracle_align_loss.argtypes = [i64, i64, i32, vp, vp, f64, i32, vp, vp, f64, f64, vp]
    lib.oracle_fold.restype = ctypes.c_int
    lib.oracle_fold.argtypes = [i64, i64, i32, vp, vp, f64, vp, i32, vp]
    lib.oracle_adapter_bytes.restype = i64
    lib.oracle_adapter_bytes.argtypes = [i32, vp, vp, i32]
    return lib


def use_library(path: str) -> None:
    """Bind this module to another build of the oracle source (the mutation
    tests load deliberately broken copies this way)."""
    global _lib
    with _lock:
        _lib = _configure(ctypes.CDLL(path))


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _configure(ctypes.CDLL(build()))
    return _lib


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _ptr_array(arrs):
    """ctypes array of pointers; keeps contiguous copies alive in the result."""
    keep = [np.ascontiguousarray(a, dtype=np.uint16) if a is not None else None for a in arrs]
    out = (ctypes.c_void_p * max(1, len(keep)))()
    for i, a in enumerate(keep):
        out[i] = a.ctypes.data if a is not None and a.size else None
    return out, keep


def apply(x, y_in, dom, slot, centroids, residuals, rows=None, gamma=None, w_base=None, w_layout=0):
    """Evaluate one projection for the listed tokens in fp64.

    x: uint16 [T, d_in] (bf16 bits); y_in: uint16 [T, d_out] or None.
    w_base: uint16 base weight, [d_in, d_out] (w_layout 0) or [d_out, d_in]
    (w_layout 1), or None; when given, x W_base is added too.
    dom, slot: int32 [T], -1 drops the term.
    gamma: float64 [T] factor on each token's centroid term, or None (1).
    centroids: list over domains of (At [rc, d_in] uint16, B [rc, d_out] uint16, s_c)
               or None for an absent domain.
    residuals: list over slots of (At [r, d_in], B [r, d_out], s_u) or None.
    rows: token indices to evaluate (default: all).
    Returns float64 [n_rows, d_out].
    """
    lib = _load()
    if w_layout not in (0, 1):
        raise ValueError(f"w_layout must be 0 ([d_in, d_out]) or 1 ([d_out, d_in]), not {w_layout!r}")
    x = np.ascontiguousarray(x, dtype=np.uint16)
    T, d_in = x.shape
    if y_in is not None:
        y_in = np.ascontiguousarray(y_in, dtype=np.uint16)
        d_out = y_in.shape[1]
    else:
        d_out = None
    dom = np.ascontiguousarray(dom, dtype=np.int32)
    slot = np.ascontiguousarray(slot, dtype=np.int32)

    def table(entries, kind_dout):
        n = len(entries)
        ranks = np.zeros(max(1, n), dtype=np.int32)
        scales = np.zeros(max(1, n), dtype=np.float64)
        ats, bs = [], []
        dout = kind_dout
        for i, e in enumerate(entries):
            if e is None:
                ats.append(None)
                bs.append(None)
                continue
            At, B, s = e
            At = np.asarray(At, dtype=np.uint16).reshape(-1, d_in)
            ranks[i] = At.shape[0]
            B = np.asarray(B, dtype=np.uint16)
            if ranks[i]:
                B = B.reshape(ranks[i], -1)
                dout = B.shape[1]
            scales[i] = float(s)
            ats.append(At)
            bs.append(B)
        pa, ka = _ptr_array(ats)
        pb, kb = _ptr_array(bs)
        return n, ranks, scales, pa, pb, (ka, kb), dout

    nd, rc, s_c, pAc, pBc, keep_c, d_out = table(centroids, d_out)
    ns, ru, s_u, pAu, pBu, keep_u, d_out = table(residuals, d_out)
    if rows is None:
        rows_arr = None
        n_rows = T
    else:
        rows_arr = np.ascontiguousarray(rows, dtype=np.int64)
        n_rows = rows_arr.shape[0]
    if w_base is not None:
        w_base = np.ascontiguousarray(w_base, dtype=np.uint16)
        if d_out is None:
            d_out = w_base.shape[1] if w_layout == 0 else w_base.shape[0]
        if w_base.shape != ((d_in, d_out) if w_layout == 0 else (d_out, d_in)):
            raise ValueError("w_base shape does not match d_in, d_out and the layout")
    if d_out is None:
        raise ValueError("cannot infer d_out: pass y_in, a factor or w_base")
    out = np.zeros((n_rows, d_out), dtype=np.float64)
    if gamma is not None:
        gamma = np.ascontiguousarray(gamma, dtype=np.float64)
        if gamma.shape != (T,):
            raise ValueError("gamma must hold one factor per token")
    rc_ = lib.oracle_apply(T, d_in, d_out, _ptr(x), _ptr(y_in) if y_in is not None else None,
                           _ptr(w_base) if w_base is not None else None, int(w_layout),
                           _ptr(dom), _ptr(slot), _ptr(gamma) if gamma is not None else None,
                           nd, _ptr(rc), _ptr(s_c), pAc, pBc,
                           ns, _ptr(ru), _ptr(s_u), pAu, pBu,
                           n_rows, _ptr(rows_arr) if rows_arr is not None else None, _ptr(out))
    if rc_ != 0:
        raise ValueError(f"oracle_apply failed with {rc_}")
    del keep_c, keep_u
    return out


def segments(dom, slot, gbin=None):
    """Grouping oracle: stable sort by (domain, gamma bin, slot), then
    maximal runs.  gbin: int32 [T] gamma bins, or None (no bins).

    Returns a dict of int32 arrays: perm, dseg_ptr, dseg_dom, dseg_gbin,
    useg_ptr, useg_dom, useg_gbin, useg_slot (each trimmed to its count).
    """
    lib = _load()
    dom = np.ascontiguousarray(dom, dtype=np.int32)
    slot = np.ascontiguousarray(slot, dtype=np.int32)
    if gbin is not None:
        gbin = np.ascontiguousarray(gbin, dtype=np.int32)
    T = dom.shape[0]
    perm = np.zeros(max(1, T), dtype=np.int32)
    dptr = np.zeros(T + 1, dtype=np.int32)
    ddom = np.zeros(max(1, T), dtype=np.int32)
    dgb = np.zeros(max(1, T), dtype=np.int32)
    uptr = np.zeros(T + 1, dtype=np.int32)
    udom = np.zeros(max(1, T), dtype=np.int32)
    ugb = np.zeros(max(1, T), dtype=np.int32)
    uslot = np.zeros(max(1, T), dtype=np.int32)
    counts = np.zeros(2, dtype=np.int32)
    rc = lib.oracle_segments(T, _ptr(dom), _ptr(gbin) if gbin is not None else None, _ptr(slot),
                             _ptr(perm), _ptr(dptr), _ptr(ddom), _ptr(dgb),
                             _ptr(uptr), _ptr(udom), _ptr(ugb), _ptr(uslot), _ptr(counts))
    if rc != 0:
        raise ValueError(f"oracle_segments failed with {rc}")
    nd, nu = int(counts[0]), int(counts[1])
    return {
        "perm": perm[:T].copy(),
        "dseg_ptr": dptr[:nd + 1].copy(),
        "dseg_dom": ddom[:nd].copy(),
        "dseg_gbin": dgb[:nd].copy(),
        "useg_ptr": uptr[:nu + 1].copy(),
        "useg_dom": udom[:nu].copy(),
        "useg_gbin": ugb[:nu].copy(),
        "useg_slot": uslot[:nu].copy(),
    }


def align_loss(At, B, s, At_c, B_c, s_c, eps=1e-8):
    """Eq. 2 from the dense matrices Delta W = s*A B and Wbar = s_c*A_c B_c.

    At [r, d_in], B [r, d_out], At_c [rc, d_in], B_c [rc, d_out]: uint16
    bf16 bits.  Returns a dict: loss, cosine, trace, norm_dw, norm_wbar.
    """
    lib = _load()
    At = np.ascontiguousarray(At, dtype=np.uint16)
    B = np.ascontiguousarray(B, dtype=np.uint16)
    At_c = np.ascontiguousarray(At_c, dtype=np.uint16)
    B_c = np.ascontiguousarray(B_c, dtype=np.uint16)
    r, d_in = At.shape
    rc = At_c.shape[0]
    d_out = B.shape[1] if r else B_c.shape[1]
    if B.shape != (r, d_out) or At_c.shape != (rc, d_in) or B_c.shape != (rc, d_out):
        raise ValueError("factor shapes do not match")
    out = np.zeros(5, dtype=np.float64)
    rc_ = lib.oracle_align_loss(d_in, d_out, r, _ptr(At), _ptr(B), float(s),
                                rc, _ptr(At_c), _ptr(B_c), float(s_c), float(eps), _ptr(out))
    if rc_ != 0:
        raise ValueError(f"oracle_align_loss failed with {rc_}")
    return {"loss": out[0], "cosine": out[1], "trace": out[2], "norm_dw": out[3], "norm_wbar": out[4]}


def fold(At_c, B_c, scale, W, layout):
    """W + scale * A_c B_c in fp64 (layout 0: W [d_in, d_out]; 1: W [d_out, d_in])."""
    lib = _load()
    At_c = np.ascontiguousarray(At_c, dtype=np.uint16)
    B_c = np.ascontiguousarray(B_c, dtype=np.uint16)
    W = np.ascontiguousarray(W, dtype=np.uint16)
    rc, d_in = At_c.shape
    d_out = B_c.shape[1]
    if W.shape != ((d_in, d_out) if layout == 0 else (d_out, d_in)):
        raise ValueError("W shape does not match the factors and layout")
    out = np.zeros(W.shape, dtype=np.float64)
    rc_ = lib.oracle_fold(d_in, d_out, rc, _ptr(At_c), _ptr(B_c), float(scale), _ptr(W), int(layout), _ptr(out))
    if rc_ != 0:
        raise ValueError(f"oracle_fold failed with {rc_}")
    return out


def adapter_bytes(d_in, d_out, rank: int) -> int:
    """Bytes of one rank-``rank`` bf16 adapter over the given weight shapes."""
    lib = _load()
    a = np.ascontiguousarray(d_in, dtype=np.int32)
    b = np.ascontiguousarray(d_out, dtype=np.int32)
    return int(lib.oracle_adapter_bytes(a.shape[0], _ptr(a), _ptr(b), rank))
