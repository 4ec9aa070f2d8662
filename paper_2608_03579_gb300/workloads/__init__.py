"""Seeded synthetic workloads for the SALT serving path.

This module draws inputs and holds none of the method's arithmetic.  Both the
fp64 oracle (tests) and the CUDA library read what it produces.  The random
numbers come from ``salt_inputs.c`` (SplitMix64 in counter mode, Box-Muller
normals rounded to bf16), so any single factor, token row or id can be
regenerated on its own, which is what lets the oracle check sampled rows of
the full-size workloads.

Recipes (shapes from the Llama-3.2-3B and Llama-3.1-8B projections; values
stand in for the paper's trained adapters and datasets, which are not used):

* x ~ N(0, 1); y_in = 0 (or N(0, 1) for the read-modify-write check)
* centroid At_c ~ N(0, 1/d_in), B_c ~ N(0, 1/rc)
* residual At_u ~ N(0, 1/d_in), B_u ~ N(0, 1/r_u)
  (the second argument of N is the variance, so each delta term is O(1))
* a token's domain is its user's slot mod n_domains
* s_c = s_u = 1 unless a test overrides them
* gamma bins: the example bins of Section "Multi-Tenant Serving",
  0.6 / 0.8 / 1.0, each token's bin uniform over them (or -1, no gamma)
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from dataclasses import dataclass, field

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "salt_inputs.c")
_LIB_PATH = os.path.join(_HERE, "libsalt_inputs.so")
_lock = threading.Lock()
_lib = None

# stream kinds (top byte of the 64-bit stream id)
K_CENT_A, K_CENT_B, K_RES_A, K_RES_B, K_X, K_Y, K_IDS, K_AUX = 1, 2, 3, 4, 5, 6, 7, 8


def build(force: bool = False) -> str:
    """Compile ``salt_inputs.c`` into ``libsalt_inputs.so`` next to it."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.run(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                    "-pthread", "-o", tmp, _SRC, "-lm"], check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            u64, i64 = ctypes.c_uint64, ctypes.c_int64
            lib.salt_inputs_bits.restype = u64
            lib.salt_inputs_bits.argtypes = [u64, u64, u64]
            lib.salt_inputs_normal_bf16.restype = None
            lib.salt_inputs_normal_bf16.argtypes = [u64, u64, u64, i64, ctypes.c_double,
                                                    ctypes.c_void_p, ctypes.c_int]
            lib.salt_inputs_uniform.restype = None
            lib.salt_inputs_uniform.argtypes = [u64, u64, u64, i64, ctypes.c_void_p]
            _lib = lib
    return _lib


def stream_id(kind: int, a: int = 0, b: int = 0, c: int = 0) -> int:
    """64-bit stream id: kind (8 bits) | a (16 bits) | b (20 bits) | c (20 bits)."""
    assert 0 <= kind < 256 and 0 <= a < (1 << 16) and 0 <= b < (1 << 20) and 0 <= c < (1 << 20)
    return (kind << 56) | (a << 40) | (b << 20) | c


def _threads() -> int:
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:  # pragma: no cover
        return os.cpu_count() or 1


def normal_bf16(seed: int, stream: int, n: int, sigma: float = 1.0, first: int = 0,
                out: np.ndarray | None = None) -> np.ndarray:
    """``n`` bf16 bit patterns of sigma * N(0, 1), elements first..first+n-1."""
    lib = _load()
    if out is None:
        out = np.empty(n, dtype=np.uint16)
    assert out.dtype == np.uint16 and out.flags.c_contiguous and out.size >= n
    if n:
        lib.salt_inputs_normal_bf16(seed, stream, first, n, float(sigma), out.ctypes.data, _threads())
    return out


def uniform(seed: int, stream: int, n: int, first: int = 0) -> np.ndarray:
    lib = _load()
    out = np.empty(n, dtype=np.float64)
    if n:
        lib.salt_inputs_uniform(seed, stream, first, n, out.ctypes.data)
    return out


def bits(seed: int, stream: int, i: int) -> int:
    return int(_load().salt_inputs_bits(seed, stream, i))


def bf16_bits_to_float(a: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def float_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest even) and return the bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def zipf_draw(u: np.ndarray, n: int, s: float = 1.1) -> np.ndarray:
    """Inverse-CDF draw from Zipf(s) truncated to {1..n}; returns ranks 1..n."""
    k = np.arange(1, n + 1, dtype=np.float64)
    p = k ** (-s)
    cdf = np.cumsum(p)
    cdf /= cdf[-1]
    r = np.searchsorted(cdf, u, side="right") + 1
    return np.minimum(r, n).astype(np.int64)


LLAMA3B_QKV = [("q_proj", 3072, 3072), ("k_proj", 3072, 1024), ("v_proj", 3072, 1024)]
LLAMA3B_MLP = [("gate_proj", 3072, 8192), ("up_proj", 3072, 8192), ("down_proj", 8192, 3072)]
LLAMA8B_LAYER = [("q_proj", 4096, 4096), ("k_proj", 4096, 1024), ("v_proj", 4096, 1024),
                 ("o_proj", 4096, 4096), ("gate_proj", 4096, 14336), ("up_proj", 4096, 14336),
                 ("down_proj", 14336, 4096)]
# adapted weight shapes behind the paper's memory columns
MISTRAL7B_QV = [("q_proj", 4096, 4096), ("v_proj", 4096, 1024)]
LLAMA3B_ALL = [("q_proj", 3072, 3072), ("k_proj", 3072, 1024), ("v_proj", 3072, 1024),
               ("o_proj", 3072, 3072), ("gate_proj", 3072, 8192), ("up_proj", 3072, 8192),
               ("down_proj", 8192, 3072)]
PYTHIA12B_ATTN = [("query_key_value", 5120, 15360), ("dense", 5120, 5120)]


@dataclass
class Workload:
    """One synthetic serving batch over a table of adapted weight matrices."""

    name: str
    seed: int
    layers: list                      # [(name, d_in, d_out)] - one entry per adapted matrix
    n_domains: int
    rc: list                          # centroid rank per domain
    n_slots: int
    r_u: list                         # residual rank per slot (0 = empty slot)
    dom_ids: np.ndarray               # int32 [T]
    slot_ids: np.ndarray              # int32 [T]
    s_c: list = field(default_factory=list)
    s_u: list = field(default_factory=list)
    y_mode: str = "zeros"             # "zeros" or "normal"
    group: list = field(default_factory=list)  # projection groups sharing one launch
    notes: str = ""

    def __post_init__(self):
        if not self.s_c:
            self.s_c = [1.0] * self.n_domains
        if not self.s_u:
            self.s_u = [1.0] * self.n_slots
        self.dom_ids = np.ascontiguousarray(self.dom_ids, dtype=np.int32)
        self.slot_ids = np.ascontiguousarray(self.slot_ids, dtype=np.int32)

    # -- shapes -----------------------------------------------------------
    @property
    def T(self) -> int:
        return int(self.dom_ids.shape[0])

    @property
    def d_in(self) -> np.ndarray:
        return np.array([l[1] for l in self.layers], dtype=np.int32)

    @property
    def d_out(self) -> np.ndarray:
        return np.array([l[2] for l in self.layers], dtype=np.int32)

    @property
    def rc_max(self) -> int:
        return max(self.rc) if self.rc else 0

    @property
    def r_max(self) -> int:
        return max(self.r_u) if self.r_u else 0

    # -- factors ------------------------------------------------------------
    def centroid_At(self, d: int, l: int) -> np.ndarray:
        r, din = self.rc[d], self.layers[l][1]
        return normal_bf16(self.seed, stream_id(K_CENT_A, d, l), r * din, 1.0 / math.sqrt(din)).reshape(r, din)

    def centroid_B(self, d: int, l: int) -> np.ndarray:
        r, dout = self.rc[d], self.layers[l][2]
        return normal_bf16(self.seed, stream_id(K_CENT_B, d, l), r * dout,
                           1.0 / math.sqrt(max(r, 1))).reshape(r, dout)

    def residual_At(self, u: int, l: int, version: int = 0, rank: int | None = None) -> np.ndarray:
        r = self.r_u[u] if rank is None else rank
        din = self.layers[l][1]
        return normal_bf16(self.seed, stream_id(K_RES_A, u, l, version), r * din,
                           1.0 / math.sqrt(din)).reshape(r, din)

    def residual_B(self, u: int, l: int, version: int = 0, rank: int | None = None) -> np.ndarray:
        r = self.r_u[u] if rank is None else rank
        dout = self.layers[l][2]
        return normal_bf16(self.seed, stream_id(K_RES_B, u, l, version), r * dout,
                           1.0 / math.sqrt(max(r, 1))).reshape(r, dout)

    def centroid_packed(self, d: int):
        """(At_all, B_all): the domain's factors over every layer, concatenated."""
        r = self.rc[d]
        din, dout = self.d_in.astype(np.int64), self.d_out.astype(np.int64)
        A = np.empty(int(r * din.sum()), dtype=np.uint16)
        B = np.empty(int(r * dout.sum()), dtype=np.uint16)
        oa = ob = 0
        for l in range(len(self.layers)):
            na, nb = int(r * din[l]), int(r * dout[l])
            normal_bf16(self.seed, stream_id(K_CENT_A, d, l), na, 1.0 / math.sqrt(din[l]), out=A[oa:oa + na])
            normal_bf16(self.seed, stream_id(K_CENT_B, d, l), nb, 1.0 / math.sqrt(max(r, 1)), out=B[ob:ob + nb])
            oa += na
            ob += nb
        return A, B

    def residual_packed(self, u: int, version: int = 0, rank: int | None = None):
        r = self.r_u[u] if rank is None else rank
        din, dout = self.d_in.astype(np.int64), self.d_out.astype(np.int64)
        A = np.empty(int(r * din.sum()), dtype=np.uint16)
        B = np.empty(int(r * dout.sum()), dtype=np.uint16)
        oa = ob = 0
        for l in range(len(self.layers)):
            na, nb = int(r * din[l]), int(r * dout[l])
            normal_bf16(self.seed, stream_id(K_RES_A, u, l, version), na, 1.0 / math.sqrt(din[l]), out=A[oa:oa + na])
            normal_bf16(self.seed, stream_id(K_RES_B, u, l, version), nb, 1.0 / math.sqrt(max(r, 1)), out=B[ob:ob + nb])
            oa += na
            ob += nb
        return A, B

    # -- activations --------------------------------------------------------
    def x(self, l: int, rows=None) -> np.ndarray:
        din = self.layers[l][1]
        if rows is None:
            return normal_bf16(self.seed, stream_id(K_X, 0, l), self.T * din).reshape(self.T, din)
        out = np.empty((len(rows), din), dtype=np.uint16)
        for i, t in enumerate(rows):
            normal_bf16(self.seed, stream_id(K_X, 0, l), din, first=int(t) * din, out=out[i])
        return out

    def y_in(self, l: int, rows=None) -> np.ndarray:
        dout = self.layers[l][2]
        n = self.T if rows is None else len(rows)
        if self.y_mode == "zeros":
            return np.zeros((n, dout), dtype=np.uint16)
        if rows is None:
            return normal_bf16(self.seed, stream_id(K_Y, 0, l), self.T * dout).reshape(self.T, dout)
        out = np.empty((len(rows), dout), dtype=np.uint16)
        for i, t in enumerate(rows):
            normal_bf16(self.seed, stream_id(K_Y, 0, l), dout, first=int(t) * dout, out=out[i])
        return out

    # -- accounting -----------------------------------------------------------
    def algorithmic_bytes(self, l: int) -> int:
        """x read, y read + write, and each distinct factor touched once."""
        din, dout = self.layers[l][1], self.layers[l][2]
        active = (self.dom_ids >= 0) | (self.slot_ids >= 0)
        n_act = int(active.sum())
        b = n_act * din * 2 + n_act * dout * 4
        for d in np.unique(self.dom_ids[self.dom_ids >= 0]):
            b += self.rc[int(d)] * (din + dout) * 2
        for u in np.unique(self.slot_ids[self.slot_ids >= 0]):
            b += self.r_u[int(u)] * (din + dout) * 2
        return int(b)

    def algorithmic_flops(self, l: int) -> int:
        din, dout = self.layers[l][1], self.layers[l][2]
        f = 0
        for d, u in zip(self.dom_ids, self.slot_ids):
            r = (self.rc[int(d)] if d >= 0 else 0) + (self.r_u[int(u)] if u >= 0 else 0)
            f += 2 * r * (din + dout)
        return int(f)


def _perm(seed: int, stream: int, n: int) -> np.ndarray:
    return np.argsort(uniform(seed, stream, n), kind="stable").astype(np.int64)


def config0(seed: int = 0) -> Workload:
    """Tiny: 512->512, 16 decode tokens in 4 user segments, 2 domains rank 8,
    4 residuals of rank 1, 2, 1, 2; token order shuffled."""
    T, users = 16, 4
    p = _perm(seed, stream_id(K_IDS, 0, 0, 0), T)
    user = (p // 4).astype(np.int32)
    return Workload("tiny", seed, [("proj", 512, 512)], 2, [8, 8], users, [1, 2, 1, 2],
                    dom_ids=user % 2, slot_ids=user, group=[[0]])


def config1(seed: int = 1) -> Workload:
    """Llama-3.2-3B decode q/k/v: 64 tokens, 4 domains rank 16, 64 users rank 2
    drawn uniformly."""
    T, n_users = 64, 64
    u = np.minimum((uniform(seed, stream_id(K_IDS, 1), T) * n_users).astype(np.int64), n_users - 1)
    return Workload("llama3b_decode_qkv", seed, list(LLAMA3B_QKV), 4, [16] * 4, n_users, [2] * n_users,
                    dom_ids=(u % 4).astype(np.int32), slot_ids=u.astype(np.int32), group=[[0, 1, 2]])


def config2(seed: int = 2) -> Workload:
    """Llama-3.2-3B prefill MLP: 8192 tokens in user segments of U{128..1024}
    tokens, 4 domains rank 32, residual ranks alternating 1 and 2."""
    T = 8192
    lens = []
    rem = T
    i = 0
    while rem > 0:
        L = 128 + int(uniform(seed, stream_id(K_IDS, 2), 1, first=i)[0] * 897)
        L = min(L, 1024)
        i += 1
        L = min(L, rem)
        lens.append(L)
        rem -= L
    if len(lens) > 1 and lens[-1] < 128:
        lens[-2] += lens[-1]
        lens.pop()
    n_users = len(lens)
    user = np.repeat(np.arange(n_users), lens).astype(np.int32)
    r_u = [1 if u % 2 == 0 else 2 for u in range(n_users)]
    return Workload("llama3b_prefill_mlp", seed, list(LLAMA3B_MLP), 4, [32] * 4, n_users, r_u,
                    dom_ids=user % 4, slot_ids=user, group=[[0, 1], [2]],
                    notes=f"segment lengths {lens}")


def config3(seed: int = 3) -> Workload:
    """Llama-3.1-8B one layer of projections, 256 decode tokens, 8 domains
    rank 64, 256 users rank 2 drawn Zipf(1.1)."""
    T, n_users = 256, 256
    k = zipf_draw(uniform(seed, stream_id(K_IDS, 3), T), n_users)
    u = (k - 1).astype(np.int32)
    return Workload("llama8b_layer_decode", seed, list(LLAMA8B_LAYER), 8, [64] * 8, n_users, [2] * n_users,
                    dom_ids=u % 8, slot_ids=u, group=[[0, 1, 2], [3], [4, 5], [6]])


# 32-layer step: slot pool regions
C4_SLOTS, C4_FIXED, C4_REGION = 512, 384, 64


def config4_region(step: int) -> int:
    """First slot of the region filled at ``step`` (alternates 384 / 448)."""
    return C4_FIXED + (step % 2) * C4_REGION


def config4_ids(seed: int, step: int, T: int = 512):
    """Token ids of one step: Zipf(1.1) over the 448 slots the step may read
    (0..383 plus the region filled in the previous step), through a fixed
    permutation; the region being filled this step is never referenced."""
    n_pos = C4_FIXED + C4_REGION
    pi = _perm(seed, stream_id(K_AUX, 4), n_pos)
    k = zipf_draw(uniform(seed, stream_id(K_IDS, 4, 0, step), T), n_pos)
    p = pi[k - 1]
    prev = config4_region(step - 1)
    slot = np.where(p < C4_FIXED, p, prev + (p - C4_FIXED)).astype(np.int32)
    return (slot % 8).astype(np.int32), slot


def config4(seed: int = 4, step: int = 1, n_layers: int = 32, T: int = 512, rank16: bool = False) -> Workload:
    """Llama-3.1-8B 32-layer stack of one layer's projections, 512 decode
    tokens, 512-slot pool, 8 domains rank 64, residuals rank 2.  With
    ``rank16`` the same step runs as standard rank-16 LoRA: no centroid,
    rank-16 adapters in the slots."""
    layers = [(f"l{i}.{n}", a, b) for i in range(n_layers) for (n, a, b) in LLAMA8B_LAYER]
    dom, slot = config4_ids(seed, step, T)
    groups = []
    for i in range(n_layers):
        b = 7 * i
        groups += [[b, b + 1, b + 2], [b + 3], [b + 4, b + 5], [b + 6]]
    if rank16:
        return Workload("llama8b_32layer_step_rank16", seed, layers, 8, [64] * 8, C4_SLOTS, [16] * C4_SLOTS,
                        dom_ids=np.full(T, -1, dtype=np.int32), slot_ids=slot, group=groups)
    return Workload("llama8b_32layer_step", seed, layers, 8, [64] * 8, C4_SLOTS, [2] * C4_SLOTS,
                    dom_ids=dom, slot_ids=slot, group=groups)


GAMMA_BINS = (0.6, 0.8, 1.0)


def gamma_bin_ids(seed: int, T: int, n_bins: int = len(GAMMA_BINS), p_none: float = 0.0) -> np.ndarray:
    """Per-token gamma bins, uniform over [0, n_bins); with probability
    p_none a token gets -1 (no gamma)."""
    g = np.minimum((uniform(seed, stream_id(K_AUX, 5), T) * n_bins).astype(np.int32), n_bins - 1)
    if p_none > 0:
        g[uniform(seed, stream_id(K_AUX, 6), T) < p_none] = -1
    return g.astype(np.int32)


CONFIGS = {0: config0, 1: config1, 2: config2, 3: config3, 4: config4}
