"""Serving-step driver over the C ABI.

Wires the four calls of a SALT serving step for a ``workloads.Workload``:
pin every domain's centroid once, pack residual blobs into page-locked host
memory and swap them into slots, group the batch, and apply the grouped
projections.  Only marshalling lives here; every step runs in libsalt.
"""
from __future__ import annotations

import numpy as np
import torch

from . import salt


def bf16_tensor(a: np.ndarray, device="cuda") -> torch.Tensor:
    """uint16 bf16 bit patterns -> torch.bfloat16 tensor on `device`."""
    t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.uint16).view(np.int16))
    return t.view(torch.bfloat16).to(device)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """torch.bfloat16 tensor -> uint16 bit patterns (host numpy)."""
    return t.detach().to("cpu").contiguous().view(torch.int16).numpy().view(np.uint16)


class SaltRunner:
    def __init__(self, wl, device: int = 0, max_tokens: int | None = None, r_max: int | None = None):
        self.wl = wl
        self.device = device
        self.d_in = wl.d_in
        self.d_out = wl.d_out
        self.r_max = r_max or max(1, wl.r_max)
        self.max_tokens = max_tokens or max(1, wl.T)
        self.ctx = salt.salt_ctx_create(self.d_in, self.d_out, wl.n_domains, max(wl.rc_max, 0), wl.n_slots,
                                        self.r_max, self.max_tokens, device)
        self.seg = salt.salt_segments_create(self.ctx)
        self._blobs = []

    def close(self):
        if self.seg:
            salt.salt_segments_destroy(self.seg)
            self.seg = None
        if self.ctx:
            salt.salt_ctx_destroy(self.ctx)
            self.ctx = None

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    # -- setup ------------------------------------------------------------
    def pin_centroids(self, scales=None):
        for d in range(self.wl.n_domains):
            if self.wl.rc[d] <= 0:
                continue
            A, B = self.wl.centroid_packed(d)
            s = self.wl.s_c[d] if scales is None else scales[d]
            salt.salt_centroid_pin(self.ctx, d, self.wl.rc[d], A, B, s)

    def blob_bytes(self, rank: int) -> int:
        return salt.salt_residual_blob_bytes(self.d_in, self.d_out, rank)

    def make_blob(self, u: int, version: int = 0, rank: int | None = None, s_u: float | None = None,
                  out: torch.Tensor | None = None) -> torch.Tensor:
        r = self.wl.r_u[u] if rank is None else rank
        A, B = self.wl.residual_packed(u, version, r)
        nb = self.blob_bytes(r)
        if out is None:
            out = torch.empty(nb, dtype=torch.uint8, pin_memory=True)
        salt.salt_residual_blob_pack(self.d_in, self.d_out, r, self.wl.s_u[u] if s_u is None else s_u,
                                     A, B, out.numpy(), nb)
        return out

    def load_slots(self, slots=None, version: int = 0, stream=None, keep: bool = False):
        """Pack and swap in the residual of each slot (synchronous per blob
        unless `keep`, which keeps every pinned blob alive)."""
        slots = range(self.wl.n_slots) if slots is None else slots
        buf = None
        for u in slots:
            if self.wl.r_u[u] <= 0:
                continue
            if keep:
                blob = self.make_blob(u, version)
                self._blobs.append(blob)
            else:
                need = self.blob_bytes(self.wl.r_u[u])
                if buf is None or buf.numel() < need:
                    buf = torch.empty(need, dtype=torch.uint8, pin_memory=True)
                blob = self.make_blob(u, version, out=buf[:need])
            salt.salt_residual_load(self.ctx, u, blob, stream)
            if not keep:
                torch.cuda.current_stream().synchronize() if stream is None else stream.synchronize()

    def build(self, dom=None, slot=None, stream=None):
        dom = self.wl.dom_ids if dom is None else dom
        slot = self.wl.slot_ids if slot is None else slot
        salt.salt_build_segments(self.ctx, self.seg, dom, slot, stream=stream)

    def alloc_xy(self, layers, zero_y: bool = False):
        xs, ys = [], []
        for l in layers:
            xs.append(bf16_tensor(self.wl.x(l)))
            ys.append(bf16_tensor(np.zeros((self.wl.T, self.d_out[l]), np.uint16) if zero_y else self.wl.y_in(l)))
        return xs, ys

    def apply(self, layers, xs, ys, stream=None):
        if len(layers) == 1:
            salt.salt_lora_apply(self.ctx, self.seg, layers[0], xs[0], ys[0], stream)
        else:
            salt.salt_lora_apply_grouped(self.ctx, self.seg, layers, xs, ys, stream)

    def device_error(self, stream=None) -> int:
        return salt.salt_get_device_error(self.ctx, stream)

    def export(self) -> dict:
        return salt.salt_segments_export(self.ctx, self.seg, self.max_tokens)
