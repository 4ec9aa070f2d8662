"""ctypes binding of ``libsalt.so`` (the C ABI in ``include/salt.h``).

Argument marshalling only: every function below forwards to the C function
of the same name; all work runs in the library's CUDA kernels.  Tensors are
passed by ``data_ptr()``; streams are ``torch.cuda.Stream`` objects (or
None for the current stream).  A non-OK status raises ``SaltError``.  If
the library has not been built, importing this module raises ImportError:
there is no fallback.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libsalt.so")

if not os.path.exists(LIB_PATH):
    raise ImportError(f"{LIB_PATH} is missing: build it with paper_2608_03579_gb300._build.build() "
                      "(nvcc, sm_103a); there is no CPU fallback")

_lib = ctypes.CDLL(LIB_PATH)

STATUS = {
    0: "SALT_OK", 1: "SALT_ERR_INVALID_ARG", 2: "SALT_ERR_OOM", 3: "SALT_ERR_NOT_PINNED_HOST",
    4: "SALT_ERR_DOMAIN_NOT_PINNED", 5: "SALT_ERR_SLOT_RANGE", 6: "SALT_ERR_RANK", 7: "SALT_ERR_LAYER_RANGE",
    8: "SALT_ERR_ALIGN", 9: "SALT_ERR_BAD_BLOB", 10: "SALT_ERR_DEVICE_IDS", 11: "SALT_ERR_TIMEOUT",
    12: "SALT_ERR_CUDA", 13: "SALT_ERR_SLOT_EMPTY", 14: "SALT_ERR_TOO_MANY_TOKENS", 15: "SALT_ERR_DOMAIN_RANGE",
    16: "SALT_ERR_STALE_SEGMENTS", 17: "SALT_ERR_NOT_BUILT", 18: "SALT_ERR_GAMMA_RANGE",
}
SALT_BLOB_HEADER_BYTES = 256
SALT_MAX_TOKENS = 16384
SALT_MAX_GROUP = 8
SALT_MAX_GAMMA_BINS = 16
SALT_MAX_RESIDUAL_RANK = 80
SALT_W_IN_OUT = 0
SALT_W_OUT_IN = 1


class SaltError(RuntimeError):
    def __init__(self, status: int, message: str = ""):
        self.status = status
        self.name = STATUS.get(status, f"status {status}")
        super().__init__(f"{self.name}: {message}" if message else self.name)


class salt_config(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_in", ctypes.POINTER(ctypes.c_int32)),
                ("d_out", ctypes.POINTER(ctypes.c_int32)), ("n_domains", ctypes.c_int32),
                ("rc_max", ctypes.c_int32), ("n_slots", ctypes.c_int32), ("r_max", ctypes.c_int32),
                ("max_tokens", ctypes.c_int32), ("device", ctypes.c_int32)]


class salt_align_pair(ctypes.Structure):
    _fields_ = [("At", ctypes.c_void_p), ("B", ctypes.c_void_p), ("At_c", ctypes.c_void_p),
                ("B_c", ctypes.c_void_p), ("r", ctypes.c_int32), ("rc", ctypes.c_int32),
                ("d_in", ctypes.c_int32), ("d_out", ctypes.c_int32), ("s", ctypes.c_float),
                ("s_c", ctypes.c_float)]


class salt_ctx_info(ctypes.Structure):
    _fields_ = [("arena_bytes", ctypes.c_int64), ("pool_bytes", ctypes.c_int64), ("slot_stride", ctypes.c_int64),
                ("apply_ctas", ctypes.c_int32), ("k_splits_max", ctypes.c_int32),
                ("apply_smem_bytes", ctypes.c_int32), ("block_tokens", ctypes.c_int32),
                ("block_users", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_vp, _i32, _i64, _f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
_SIGS = {
    "salt_abi_version": (_i32, []),
    "salt_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "salt_ctx_create": (ctypes.c_int, [ctypes.POINTER(salt_config), ctypes.POINTER(_vp)]),
    "salt_ctx_destroy": (None, [_vp]),
    "salt_last_error": (ctypes.c_char_p, [_vp]),
    "salt_ctx_get_info": (ctypes.c_int, [_vp, ctypes.POINTER(salt_ctx_info)]),
    "salt_centroid_pin": (ctypes.c_int, [_vp, _i32, _i32, _vp, _vp, _f32]),
    "salt_residual_blob_bytes": (_i64, [ctypes.POINTER(salt_config), _i32]),
    "salt_residual_blob_pack": (ctypes.c_int, [ctypes.POINTER(salt_config), _i32, _f32, _vp, _vp, _vp, _i64]),
    "salt_residual_load": (ctypes.c_int, [_vp, _i32, _vp, _vp]),
    "salt_residual_load_batch": (ctypes.c_int, [_vp, _i32, _vp, _vp, _vp]),
    "salt_segments_create": (ctypes.c_int, [_vp, ctypes.POINTER(_vp)]),
    "salt_segments_destroy": (None, [_vp]),
    "salt_build_segments": (ctypes.c_int, [_vp, _vp, _vp, _vp, _i32, _vp]),
    "salt_segments_export": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp]),
    "salt_lora_apply": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp, _vp]),
    "salt_lora_apply_grouped": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp, _vp, _vp]),
    "salt_lora_apply_static": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp, _vp]),
    "salt_get_device_error": (ctypes.c_int, [_vp, _vp, ctypes.POINTER(ctypes.c_uint32)]),
    "salt_selftest_wait_timeout": (ctypes.c_int, [_vp, _vp]),
    "salt_host_alloc": (_vp, [_i64]),
    "salt_host_free": (None, [_vp]),
    "salt_residual_blob_concat": (ctypes.c_int, [ctypes.POINTER(salt_config), _i32, _vp, _vp, _f32, _i32, _vp, _vp,
                                                 _f32, _vp, _i64]),
    "salt_centroid_fold": (ctypes.c_int, [_vp, _i32, _i32, _f32, _vp, _i32, _vp]),
    "salt_build_segments_gamma": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _vp]),
    "salt_segments_export_gamma": (ctypes.c_int, [_vp, _vp, _vp, _vp]),
    "salt_align_loss": (ctypes.c_int, [_i32, ctypes.POINTER(salt_align_pair), _f32, _vp, _vp, _vp]),
    "salt_host_pipe_create": (ctypes.c_int, [_vp, _i32, _i64, ctypes.POINTER(_vp)]),
    "salt_host_pipe_destroy": (None, [_vp]),
    "salt_lora_apply_host": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp, _vp, _vp]),
    "salt_host_pipe_wait": (ctypes.c_int, [_vp, _vp]),
    "salt_guard_check": (ctypes.c_int, [_vp, _vp, ctypes.POINTER(ctypes.c_int32)]),
    "salt_lora_apply_with_base": (ctypes.c_int, [_vp, _vp, _i32, _vp, _vp, _i32, _vp, _vp]),
    "salt_fold_plan_create": (ctypes.c_int, [_vp, _i32, _i32, _vp, _vp, _i32, ctypes.POINTER(_vp)]),
    "salt_fold_plan_run": (ctypes.c_int, [_vp, _f32, _vp]),
    "salt_fold_plan_destroy": (None, [_vp]),
}
for _name, (_res, _args) in _SIGS.items():
    _f = getattr(_lib, _name)
    _f.restype = _res
    _f.argtypes = _args


def _check(status: int, ctx=None):
    if status != 0:
        msg = _lib.salt_last_error(ctx).decode() if ctx else ""
        raise SaltError(status, msg)


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(a) -> int | None:
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        assert a.flags.c_contiguous
        return a.ctypes.data
    if isinstance(a, int):
        return a
    assert a.is_contiguous()
    return a.data_ptr()


def make_config(d_in, d_out, n_domains=0, rc_max=0, n_slots=0, r_max=1, max_tokens=1, device=0):
    """A salt_config plus the arrays it points to (kept alive on the object)."""
    din = np.ascontiguousarray(d_in, dtype=np.int32)
    dout = np.ascontiguousarray(d_out, dtype=np.int32)
    c = salt_config(len(din), din.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)),
                    dout.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), n_domains, rc_max, n_slots, r_max,
                    max_tokens, device)
    c._keep = (din, dout)
    return c


def salt_abi_version() -> int:
    return int(_lib.salt_abi_version())


def salt_status_string(status: int) -> str:
    return _lib.salt_status_string(status).decode()


def salt_ctx_create(d_in, d_out, n_domains, rc_max, n_slots, r_max, max_tokens, device=0) -> int:
    cfg = make_config(d_in, d_out, n_domains, rc_max, n_slots, r_max, max_tokens, device)
    out = _vp()
    _check(_lib.salt_ctx_create(ctypes.byref(cfg), ctypes.byref(out)))
    return out.value


def salt_ctx_destroy(ctx) -> None:
    _lib.salt_ctx_destroy(ctx)


def salt_last_error(ctx) -> str:
    return _lib.salt_last_error(ctx).decode()


def salt_ctx_get_info(ctx) -> dict:
    info = salt_ctx_info()
    _check(_lib.salt_ctx_get_info(ctx, ctypes.byref(info)), ctx)
    return {k: getattr(info, k) for (k, _) in salt_ctx_info._fields_ if k != "reserved"}


def salt_centroid_pin(ctx, domain: int, rc: int, At_c, B_c, s_c: float) -> None:
    _check(_lib.salt_centroid_pin(ctx, domain, rc, _ptr(At_c), _ptr(B_c), float(s_c)), ctx)


def salt_residual_blob_bytes(d_in, d_out, rank: int) -> int:
    return int(_lib.salt_residual_blob_bytes(ctypes.byref(make_config(d_in, d_out)), rank))


def salt_residual_blob_pack(d_in, d_out, rank: int, s_u: float, At_u, B_u, blob, blob_bytes: int) -> None:
    cfg = make_config(d_in, d_out)
    _check(_lib.salt_residual_blob_pack(ctypes.byref(cfg), rank, float(s_u), _ptr(At_u), _ptr(B_u),
                                        _ptr(blob), blob_bytes))


def salt_residual_blob_concat(d_in, d_out, rc: int, At_c, B_c, s_c: float, rank: int, At_u, B_u, s_u: float,
                              blob, blob_bytes: int) -> None:
    """Blob of rank rc + rank holding the scaled centroid and the residual as
    one ordinary adapter (the long-tail form)."""
    cfg = make_config(d_in, d_out)
    _check(_lib.salt_residual_blob_concat(ctypes.byref(cfg), rc, _ptr(At_c), _ptr(B_c), float(s_c), rank,
                                          _ptr(At_u), _ptr(B_u), float(s_u), _ptr(blob), blob_bytes))


def salt_centroid_fold(ctx, domain: int, layer: int, gamma: float, W, layout: int = SALT_W_IN_OUT,
                       stream=None) -> None:
    """W += gamma * s_c(domain) * A_c B_c in place (W a CUDA bf16 tensor)."""
    _check(_lib.salt_centroid_fold(ctx, domain, layer, float(gamma), _ptr(W), layout, _stream(stream)), ctx)


class FoldPlan:
    """A salt_fold_plan handle; keeps the weight tensors alive with it."""

    def __init__(self, ctx, handle, weights):
        self.ctx, self.handle, self._weights = ctx, handle, weights


def salt_fold_plan_create(ctx, domain: int, layers, weights, layout: int = SALT_W_IN_OUT) -> FoldPlan:
    """One launch that folds domain's centroid into every weight (CUDA bf16
    tensors) of `weights`, weights[i] being layer layers[i]'s."""
    n = len(layers)
    if len(weights) != n:
        raise ValueError("one weight per layer")
    ls = (ctypes.c_int32 * max(1, n))(*[int(l) for l in layers])
    ws = (_vp * max(1, n))(*[_ptr(w) for w in weights])
    h = _vp()
    _check(_lib.salt_fold_plan_create(ctx, int(domain), n, ls, ws, int(layout), ctypes.byref(h)), ctx)
    return FoldPlan(ctx, h, list(weights))


def salt_fold_plan_run(plan: FoldPlan, gamma: float, stream=None) -> None:
    _check(_lib.salt_fold_plan_run(plan.handle, float(gamma), _stream(stream)), plan.ctx)


def salt_fold_plan_destroy(plan: FoldPlan) -> None:
    if plan is not None and plan.handle:
        _lib.salt_fold_plan_destroy(plan.handle)
        plan.handle = None


def salt_align_pairs(pairs):
    """The C array of salt_align_pair for a sequence of dicts with At, B,
    At_c, B_c (CUDA bf16 tensors or device addresses), r, rc, d_in, d_out,
    s, s_c; reusable across calls while the tensors live."""
    arr = (salt_align_pair * max(1, len(pairs)))()
    for i, q in enumerate(pairs):
        arr[i] = salt_align_pair(_ptr(q["At"]), _ptr(q["B"]), _ptr(q["At_c"]), _ptr(q["B_c"]), int(q["r"]),
                                 int(q["rc"]), int(q["d_in"]), int(q["d_out"]), float(q["s"]), float(q["s_c"]))
    arr._n = len(pairs)
    return arr


def salt_align_loss(pairs, eps: float, loss, cosine=None, stream=None) -> None:
    """pairs: a sequence of dicts (see salt_align_pairs) or its prepared
    array.  loss / cosine: CUDA float32 tensors of len(pairs) (cosine may be
    None)."""
    arr = pairs if hasattr(pairs, "_n") else salt_align_pairs(pairs)
    _check(_lib.salt_align_loss(arr._n, arr, float(eps), _ptr(loss), _ptr(cosine), _stream(stream)))


class HostBuffer:
    """Huge-page-backed page-locked host memory from salt_host_alloc, viewed
    as a uint8 torch tensor (``.tensor``); freed by ``close()`` or on
    garbage collection."""

    def __init__(self, nbytes: int):
        import torch
        self.ptr = _lib.salt_host_alloc(int(nbytes))
        if not self.ptr:
            raise SaltError(2, f"salt_host_alloc({nbytes}) failed")
        self.nbytes = int(nbytes)
        arr = np.ctypeslib.as_array((ctypes.c_uint8 * self.nbytes).from_address(self.ptr))
        self.tensor = torch.from_numpy(arr)

    def close(self):
        if self.ptr:
            self.tensor = None
            _lib.salt_host_free(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def salt_host_alloc(nbytes: int) -> HostBuffer:
    return HostBuffer(nbytes)


def salt_host_free(buf) -> None:
    """Release a HostBuffer (or a raw pointer from the C call)."""
    if isinstance(buf, HostBuffer):
        buf.close()
    elif buf:
        _lib.salt_host_free(buf)


def salt_residual_load(ctx, slot: int, host_blob, stream=None) -> None:
    _check(_lib.salt_residual_load(ctx, slot, _ptr(host_blob), _stream(stream)), ctx)


def salt_residual_load_batch(ctx, slots, host_blobs, stream=None) -> None:
    """The loads of salt_residual_load for each (slot, blob) pair, in one call."""
    n = len(slots)
    if len(host_blobs) != n:
        raise ValueError("one blob per slot")
    sl = (_i32 * max(n, 1))(*[int(x) for x in slots])
    bl = (_vp * max(n, 1))(*[_ptr(b) for b in host_blobs])
    _check(_lib.salt_residual_load_batch(ctx, n, sl, bl, _stream(stream)), ctx)


def salt_segments_create(ctx) -> int:
    out = _vp()
    _check(_lib.salt_segments_create(ctx, ctypes.byref(out)), ctx)
    return out.value


def salt_segments_destroy(seg) -> None:
    _lib.salt_segments_destroy(seg)


def salt_build_segments(ctx, seg, domain_ids, slot_ids, n_tokens: int | None = None, stream=None) -> None:
    """ids: numpy / CPU tensors (host path) or CUDA int32 tensors (device path)."""
    if isinstance(domain_ids, np.ndarray):
        domain_ids = np.ascontiguousarray(domain_ids, dtype=np.int32)
        slot_ids = np.ascontiguousarray(slot_ids, dtype=np.int32)
    n = len(domain_ids) if n_tokens is None else n_tokens
    _check(_lib.salt_build_segments(ctx, seg, _ptr(domain_ids), _ptr(slot_ids), n, _stream(stream)), ctx)


def salt_build_segments_gamma(ctx, seg, domain_ids, gamma_bins, slot_ids, gamma, n_tokens: int | None = None,
                              stream=None) -> None:
    """salt_build_segments with per-token gamma bins; gamma: the bins' values."""
    if isinstance(domain_ids, np.ndarray):
        domain_ids = np.ascontiguousarray(domain_ids, dtype=np.int32)
        slot_ids = np.ascontiguousarray(slot_ids, dtype=np.int32)
    if isinstance(gamma_bins, np.ndarray):
        gamma_bins = np.ascontiguousarray(gamma_bins, dtype=np.int32)
    g = np.ascontiguousarray(gamma, dtype=np.float32)
    n = len(domain_ids) if n_tokens is None else n_tokens
    _check(_lib.salt_build_segments_gamma(ctx, seg, _ptr(domain_ids), _ptr(gamma_bins), _ptr(slot_ids), n,
                                          len(g), g.ctypes.data if len(g) else None, _stream(stream)), ctx)


def salt_segments_export_gamma(ctx, seg, max_tokens: int) -> dict:
    """The gamma bins of the domain runs and user runs of the last build."""
    counts = salt_segments_export(ctx, seg, max_tokens)["counts"]
    dg = np.zeros(max_tokens + 1, dtype=np.int32)
    ug = np.zeros(max_tokens + 1, dtype=np.int32)
    _check(_lib.salt_segments_export_gamma(ctx, seg, dg.ctypes.data, ug.ctypes.data), ctx)
    return {"dseg_gbin": dg[:int(counts[1])], "useg_gbin": ug[:int(counts[2])]}


def salt_segments_export(ctx, seg, max_tokens: int) -> dict:
    n = max_tokens + 1
    counts = np.zeros(4, dtype=np.int32)
    arrs = {k: np.zeros(n, dtype=np.int32) for k in
            ("perm", "dseg_ptr", "dseg_dom", "useg_ptr", "useg_dom", "useg_slot")}
    blocks = np.zeros(3 * n, dtype=np.int32)
    _check(_lib.salt_segments_export(ctx, seg, counts.ctypes.data, arrs["perm"].ctypes.data,
                                     arrs["dseg_ptr"].ctypes.data, arrs["dseg_dom"].ctypes.data,
                                     arrs["useg_ptr"].ctypes.data, arrs["useg_dom"].ctypes.data,
                                     arrs["useg_slot"].ctypes.data, blocks.ctypes.data), ctx)
    T, nd, nu, nb = (int(v) for v in counts)
    return {"perm": arrs["perm"][:T], "dseg_ptr": arrs["dseg_ptr"][:nd + 1], "dseg_dom": arrs["dseg_dom"][:nd],
            "useg_ptr": arrs["useg_ptr"][:nu + 1], "useg_dom": arrs["useg_dom"][:nu],
            "useg_slot": arrs["useg_slot"][:nu], "blocks": blocks[:3 * nb].reshape(nb, 3), "counts": counts}


def salt_lora_apply(ctx, seg, layer: int, x, y, stream=None) -> None:
    _check(_lib.salt_lora_apply(ctx, seg, layer, _ptr(x), _ptr(y), _stream(stream)), ctx)


def salt_lora_apply_with_base(ctx, seg, layer: int, x, W, layout: int, y, stream=None) -> None:
    """y = x W_base + the SALT delta (y written, not read)."""
    _check(_lib.salt_lora_apply_with_base(ctx, seg, layer, _ptr(x), _ptr(W), layout, _ptr(y), _stream(stream)), ctx)


def salt_lora_apply_static(ctx, seg, layer: int, x, y, stream=None) -> None:
    """salt_lora_apply without any device allocation behind it (static scratch)."""
    _check(_lib.salt_lora_apply_static(ctx, seg, layer, _ptr(x), _ptr(y), _stream(stream)), ctx)


def salt_lora_apply_grouped(ctx, seg, layers, xs, ys, stream=None) -> None:
    n = len(layers)
    la = (ctypes.c_int32 * n)(*layers)
    xa = (ctypes.c_void_p * n)(*[_ptr(t) for t in xs])
    ya = (ctypes.c_void_p * n)(*[_ptr(t) for t in ys])
    _check(_lib.salt_lora_apply_grouped(ctx, seg, n, la, xa, ya, _stream(stream)), ctx)


class HostPipe:
    """A salt_host_pipe handle with the context it belongs to (for error messages)."""

    def __init__(self, ctx, n_stages: int = 0, stage_bytes: int = 0):
        out = _vp()
        _check(_lib.salt_host_pipe_create(ctx, n_stages, stage_bytes, ctypes.byref(out)), ctx)
        self.ctx, self.ptr = ctx, out.value

    def close(self):
        if self.ptr:
            _lib.salt_host_pipe_destroy(self.ptr)
            self.ptr = None


def salt_host_pipe_create(ctx, n_stages: int = 0, stage_bytes: int = 0) -> HostPipe:
    return HostPipe(ctx, n_stages, stage_bytes)


def salt_host_pipe_destroy(pipe) -> None:
    pipe.close()


def salt_lora_apply_host(pipe, seg, layers, x_hosts, y_hosts, stream=None) -> None:
    """Grouped apply on page-locked host activations (copies in, apply, copies out)."""
    n = len(layers)
    la = (ctypes.c_int32 * n)(*layers)
    xa = (ctypes.c_void_p * n)(*[_ptr(t) for t in x_hosts])
    ya = (ctypes.c_void_p * n)(*[_ptr(t) for t in y_hosts])
    _check(_lib.salt_lora_apply_host(pipe.ptr, seg, n, la, xa, ya, _stream(stream)), pipe.ctx)


def salt_host_pipe_wait(pipe, stream=None) -> None:
    _check(_lib.salt_host_pipe_wait(pipe.ptr, _stream(stream)), pipe.ctx)


def salt_guard_check(ctx, seg=None) -> int:
    """Number of damaged guard bands around the library's device buffers (synchronous)."""
    n = ctypes.c_int32(0)
    _check(_lib.salt_guard_check(ctx, seg, ctypes.byref(n)), ctx)
    return int(n.value)


def salt_selftest_wait_timeout(ctx, stream=None) -> None:
    _check(_lib.salt_selftest_wait_timeout(ctx, _stream(stream)), ctx)


def salt_get_device_error(ctx, stream=None, raise_on_flags: bool = False) -> int:
    flags = ctypes.c_uint32(0)
    st = _lib.salt_get_device_error(ctx, _stream(stream), ctypes.byref(flags))
    if st not in (0, 10) or (raise_on_flags and st == 10):
        _check(st, ctx)
    return int(flags.value)
