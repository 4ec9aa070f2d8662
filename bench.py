"""Benchmark of the SALT serving hot path on GB300.

One step = one pass of the whole per-step path over one decode batch of the
Llama-3.1-8B 32-layer workload (512 tokens, 8 domains with rank-64
centroids, a 512-slot pool of rank-2 residuals drawn Zipf(1.1)):

  1. 64 new residual blobs are swapped host -> device into the slot region
     the batch does not read, on a side stream (salt_residual_load),
  2. the batch is grouped (salt_build_segments, host ids),
  3. every adapted projection of the 32 layers is applied in place
     (salt_lora_apply_grouped: q/k/v, o, gate/up, down per layer; 128
     launches replayed from one CUDA graph).

The swaps overlap the applies (the paper's swap-light serving).  Inputs are
synthetic, drawn by the seeded generator; nothing comes from a dataset or a
trained checkpoint.  `value` is tokens/s with x / y resident in HBM; `e2e`
adds the host <-> device copies of x, y_in and y to every step.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--mode salt|rank16]
                  [--gamma-bins] [--row fold|align]

--gamma-bins groups the same step by (centroid, gamma bin), each token in
one of the bins 0.6 / 0.8 / 1.0 (salt_build_segments_gamma).  --row prints
the line of another part of the path instead of the step: `fold` fuses one
domain's rank-64 centroid into all 224 adapted weights of the 32 layers
(salt_centroid_fold, alternating +gamma and -gamma), `align` evaluates the
alignment regulariser over the same 224 matrices for a rank-16 task update
against the rank-64 centroid (salt_align_loss).

Under torchrun (N > 1) every rank runs an independent replica on its own
GPU (the path has no exchange step); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "centroid+residual LoRA apply tokens/s; achieved HBM GB/s as % of GB300 peak"
WORKLOAD = "llama8b_32layer_decode_step"
PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0}


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="salt", choices=["salt", "reference"])
    ap.add_argument("--mode", default="salt", choices=["salt", "rank16"])
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--gamma-bins", action="store_true")
    ap.add_argument("--row", default="step", choices=["step", "fold", "align", "base"])
    ap.add_argument("--config", type=int, default=4, choices=[1, 2, 3, 4],
                    help="4: the 32-layer decode step (default); 1-3: the other serving configurations")
    ap.add_argument("--clocks-csv", default=None, help="also write the raw nvidia-smi samples of the timed region here")
    return ap.parse_args()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return dict(PEAKS_FALLBACK), "fallback"


# ----------------------------------------------------------------------------- distributed
def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    pg = None
    if world > 1:
        import torch.distributed as dist
        import torch
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
        pg = dist
    return rank, world, local, pg


def barrier(pg, device=None):
    if pg is not None:
        import torch
        if device is not None and pg.get_backend() == "nccl":
            pg.barrier(device_ids=[device])
        else:
            pg.barrier()


def max_over_ranks(pg, v: float, device=None) -> float:
    if pg is None:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64, device=f"cuda:{device}" if pg.get_backend() == "nccl" else "cpu")
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi sampling of SM clock and throttle reasons during a region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_uuid: str | None, out_path: str | None = None):
        self.uuid = gpu_uuid
        self.proc = None
        self.lines = []
        self.out_path = out_path

    def __enter__(self):
        cmd = ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200"]
        if self.uuid:
            cmd += ["-i", self.uuid]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=2)
        if self.out_path and self.lines:
            with open(self.out_path, "w") as f:
                f.write(self.FIELDS + "\n" + "\n".join(self.lines) + "\n")

    def summary(self):
        mhz, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                mhz.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not mhz:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(mhz)}


# ----------------------------------------------------------------------------- workload setup
def groups_of(n_layers):
    g = []
    for i in range(n_layers):
        b = 7 * i
        g += [[b, b + 1, b + 2], [b + 3], [b + 4, b + 5], [b + 6]]
    return g


class Step:
    """Device state and per-step actions of the 32-layer decode step."""

    N_ID_SETS = 8

    def __init__(self, args, device: int):
        import torch
        from paper_2608_03579_gb300 import workloads as wl
        from paper_2608_03579_gb300 import salt
        from paper_2608_03579_gb300.runner import SaltRunner

        self.torch, self.salt, self.wl_mod = torch, salt, wl
        self.device = device
        rank16 = args.mode == "rank16"
        self.rank16 = rank16
        self.w = wl.config4(seed=4, step=1, n_layers=args.layers, rank16=rank16)
        self.T = self.w.T
        self.L = len(self.w.layers)
        self.groups = groups_of(args.layers)
        self.ids = [wl.config4_ids(4, s, self.T) for s in range(self.N_ID_SETS)]
        self.gbins = ([wl.gamma_bin_ids(4 + s, self.T) for s in range(self.N_ID_SETS)]
                      if getattr(args, "gamma_bins", False) else None)
        if rank16:
            self.ids = [(np.full(self.T, -1, np.int32), sl) for (_, sl) in self.ids]
        self.runner = SaltRunner(self.w, device=device, max_tokens=self.T)
        r = self.runner
        if not rank16:
            r.pin_centroids()
        # initial fill of the whole pool; rank-16 mode reuses 64 distinct blobs.
        # The blobs a step swaps in live in one huge-page-backed page-locked
        # region (salt_host_alloc), as a serving engine's host-side residual
        # cache would.
        r_slot = 16 if rank16 else 2
        nb = r.blob_bytes(r_slot)
        pitch = (nb + 255) // 256 * 256
        n_host = 64 if rank16 else 2 * wl.C4_REGION
        self.host_buf = salt.salt_host_alloc(n_host * pitch)
        self.host_huge = huge_page_bytes(self.host_buf.ptr)
        blob_at = lambda k: self.host_buf.tensor[k * pitch:k * pitch + nb]
        if rank16:
            base = [r.make_blob(u, 0, r_slot, out=blob_at(u)) for u in range(64)]
            for u in range(self.w.n_slots):
                salt.salt_residual_load(r.ctx, u, base[u % 64], None)
            torch.cuda.synchronize()
            self.host_sets = [base, base]
        else:
            r.load_slots()
            self.host_sets = [[r.make_blob(wl.config4_region(p) + i, 1 + p, out=blob_at(p * wl.C4_REGION + i))
                               for i in range(wl.C4_REGION)] for p in range(2)]
        self.blob_bytes = nb
        # activations: one contiguous buffer for all projections
        self.x_off, self.y_off = [], []
        xo = yo = 0
        for (_, din, dout) in self.w.layers:
            self.x_off.append(xo)
            self.y_off.append(yo)
            xo += self.T * din
            yo += self.T * dout
        self.x_elems, self.y_elems = xo, yo
        self.x_all = torch.empty(xo, dtype=torch.bfloat16, device=f"cuda:{device}")
        self.y_all = torch.zeros(yo, dtype=torch.bfloat16, device=f"cuda:{device}")
        xh = np.empty(xo, dtype=np.uint16)
        for l in range(self.L):
            din = self.w.layers[l][1]
            wl.normal_bf16(self.w.seed, wl.stream_id(wl.K_X, 0, l), self.T * din,
                           out=xh[self.x_off[l]:self.x_off[l] + self.T * din])
        self.x_all.copy_(torch.from_numpy(xh.view(np.int16)).view(torch.bfloat16))
        self.xs = [self.x_all[self.x_off[l]:self.x_off[l] + self.T * self.w.layers[l][1]] for l in range(self.L)]
        self.ys = [self.y_all[self.y_off[l]:self.y_off[l] + self.T * self.w.layers[l][2]] for l in range(self.L)]
        self.comp = torch.cuda.Stream(device=device)
        self.side = torch.cuda.Stream(device=device)
        self.graph = None

    # one step's actions
    def swap(self, s):
        region = self.wl_mod.config4_region(s % self.N_ID_SETS)
        hs = self.host_sets[s % 2]
        n = self.wl_mod.C4_REGION
        self.salt.salt_residual_load_batch(self.runner.ctx, list(range(region, region + n)), hs[:n], self.side)

    def build(self, s):
        dom, slot = self.ids[s % self.N_ID_SETS]
        if self.gbins is not None:
            self.salt.salt_build_segments_gamma(self.runner.ctx, self.runner.seg, dom, self.gbins[s % self.N_ID_SETS],
                                                slot, self.wl_mod.GAMMA_BINS, stream=self.comp)
        else:
            self.salt.salt_build_segments(self.runner.ctx, self.runner.seg, dom, slot, stream=self.comp)

    def applies_eager(self, timing=False):
        torch = self.torch
        evs = []
        with torch.cuda.stream(self.comp):
            for grp in self.groups:
                if timing:
                    a = torch.cuda.Event(enable_timing=True)
                    b = torch.cuda.Event(enable_timing=True)
                    a.record()
                self.salt.salt_lora_apply_grouped(self.runner.ctx, self.runner.seg, grp,
                                                  [self.xs[l] for l in grp], [self.ys[l] for l in grp], self.comp)
                if timing:
                    b.record()
                    evs.append((a, b))
        return evs

    def capture(self):
        """One CUDA graph of the 128 grouped applies of a step."""
        torch = self.torch
        self.build(0)
        self.applies_eager()
        torch.cuda.synchronize(self.device)
        g = torch.cuda.CUDAGraph()
        try:
            with torch.cuda.graph(g, stream=self.comp):
                for grp in self.groups:
                    self.salt.salt_lora_apply_grouped(self.runner.ctx, self.runner.seg, grp,
                                                      [self.xs[l] for l in grp], [self.ys[l] for l in grp],
                                                      self.comp)
            self.graph = g
        except Exception as e:  # graph capture unavailable: eager launches
            print(f"graph capture failed ({e}); using eager launches", file=sys.stderr)
            torch.cuda.synchronize(self.device)
            self.graph = None

    def applies(self):
        if self.graph is not None:
            with self.torch.cuda.stream(self.comp):
                self.graph.replay()
            return []
        return self.applies_eager()

    def step(self, s, timing=False):
        """One whole step; with `timing`, the applies are launched eagerly with a
        CUDA event pair around each launch (returned)."""
        self.swap(s)
        self.build(s)
        if timing:
            return self.applies_eager(timing=True)
        return self.applies()

    def join_side(self):
        self.comp.wait_stream(self.side)

    def apply_bytes(self):
        """Algorithmic bytes of one step's applies, per launch group, averaged over the id sets."""
        per_group = np.zeros(len(self.groups))
        for dom, slot in self.ids:
            w = self.w
            w.dom_ids, w.slot_ids = dom, slot
            for gi, grp in enumerate(self.groups):
                per_group[gi] += sum(w.algorithmic_bytes(l) for l in grp)
        return per_group / len(self.ids)

    def close(self):
        self.graph = None
        self.runner.close()
        self.host_sets = None
        self.host_buf.close()


# ----------------------------------------------------------------------------- oracle timing
def host_cores() -> int:
    """Cores this process may run on (its affinity mask)."""
    try:
        return len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        return os.cpu_count() or 1


class OracleSampler:
    """The fp64 oracle on a bounded sample of the step: some of the 512
    tokens of one of the 32 layers, all 7 projections, with the tables of
    that layer built once.  With n threads the tokens are split into n
    disjoint slices, each evaluated by the same oracle call on its own host
    thread (the C oracle runs outside the interpreter lock), so the oracle's
    arithmetic is unchanged; only the tokens are shared out."""

    def __init__(self, mode: str, n_layers: int):
        import oracle
        from paper_2608_03579_gb300 import workloads as wl
        oracle.build()
        self.oracle = oracle
        w = wl.config4(seed=4, step=1, n_layers=1, rank16=(mode == "rank16"))
        self.T, self.n_layers, self.mode = w.T, n_layers, mode
        self.dom = w.dom_ids if mode != "rank16" else np.full(w.T, -1, np.int32)
        self.slot = w.slot_ids
        used = set(int(s) for s in w.slot_ids if s >= 0)
        self.tables = []
        for l in range(7):
            cents = ([(w.centroid_At(d, l), w.centroid_B(d, l), 1.0) for d in range(w.n_domains)]
                     if mode != "rank16" else [])
            res = [((w.residual_At(u, l), w.residual_B(u, l), 1.0) if u in used else None)
                   for u in range(w.n_slots)]
            self.tables.append((w.x(l), w.y_in(l), cents, res))

    def rows(self, n: int) -> np.ndarray:
        """n tokens spread evenly over the batch (its domain and user mix)."""
        n = max(1, min(n, self.T))
        return np.unique(np.linspace(0, self.T - 1, n).round().astype(np.int64))

    def run(self, n_tokens: int, threads: int = 1, repeat: int = 1):
        """Seconds to evaluate n_tokens tokens of one layer `repeat` times on
        `threads` threads; returns (seconds, token-layers evaluated)."""
        rows = self.rows(n_tokens)
        parts = [p for p in np.array_split(rows, max(1, min(threads, len(rows)))) if len(p)]

        def work(part):
            for _ in range(repeat):
                for (x, y, cents, res) in self.tables:
                    self.oracle.apply(x, y, self.dom, self.slot, cents, res, rows=part)

        t0 = time.perf_counter()
        if len(parts) == 1:
            work(parts[0])
        else:
            ts = [threading.Thread(target=work, args=(p,)) for p in parts]
            for t in ts:
                t.start()
            for t in ts:
                t.join()
        return time.perf_counter() - t0, len(rows) * repeat

    def tokens_per_s(self, seconds: float, token_layers: int) -> float:
        """Whole-step tokens/s: a token of the step passes all n_layers layers."""
        return token_layers / self.n_layers / seconds

    def sized(self, seconds_target: float, threads: int):
        """(tokens, repeat) that take about seconds_target on `threads` threads:
        up to the whole batch of one layer, then that layer repeated."""
        dt, n = self.run(4 * threads, threads)
        wall_per_token = dt / n
        want = max(threads, int(seconds_target / max(wall_per_token, 1e-9)))
        if want <= self.T:
            return want, 1
        return self.T, max(1, round(want / self.T))


def cpu_baseline_line(mode: str, n_layers: int, seconds: float) -> dict:
    """The oracle timed on the host cores, single-threaded and on every core
    of the affinity mask; `value` and `cores` are the all-core run's."""
    smp = OracleSampler(mode, n_layers)
    cores = host_cores()
    out = {}
    for th in sorted({1, cores}):
        n, rep = smp.sized(seconds / 2, th)
        dt, tl = smp.run(n, th, rep)
        out[th] = (smp.tokens_per_s(dt, tl), n, rep, dt)
    v1, n1, r1, d1 = out[1]
    vn, nn, rn, dn = out[cores]
    return {"value": vn, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": (f"{nn} of the 512 tokens x the 7 projections of 1 of {n_layers} layers, x{rn}, on {cores} "
                       f"threads ({dn:.1f} s); tokens/s = token-layers / {n_layers} / seconds; fp64 C oracle, "
                       f"tokens split over threads"),
            "single_thread": {"value": v1, "unit": "tokens/s", "cores": 1,
                              "sample": f"{n1} tokens x 7 projections x 1 layer, x{r1} ({d1:.1f} s)"},
            "cores_source": "os.sched_getaffinity"}


# ----------------------------------------------------------------------------- main arms
def run_reference(args, rank, world, pg):
    """The oracle arm: the fp64 CPU oracle timed on the host cores of rank 0.

    Each step evaluates a bounded sample of the step (tokens of one of the 32
    layers, all 7 projections) on every core; the line reports the steps it
    ran, the seconds they took and the tokens they processed, and converts
    them to whole-step tokens/s (a token of the step passes all 32 layers)."""
    if rank != 0:
        return
    smp = OracleSampler(args.mode, args.layers)
    cores = host_cores()
    n_tok, rep = smp.sized(2.0, cores)  # about 2 s a step on every core
    for _ in range(args.warmup):
        smp.run(max(cores, n_tok // 8), cores)
    secs, toks = [], 0
    for _ in range(args.steps):
        dt, n = smp.run(n_tok, cores, rep)
        secs.append(dt)
        toks += n
    total = float(sum(secs))
    value = toks / args.layers / total
    d1, n1 = smp.run(max(1, n_tok // cores), 1)
    v1 = smp.tokens_per_s(d1, n1)
    sample = (f"each step: {n_tok} of the 512 tokens x the 7 projections of 1 of {args.layers} layers, x{rep}, "
              f"on {cores} threads; tokens/s = token-layers evaluated / {args.layers} / seconds")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": WORKLOAD, "tokens_per_step": 512, "layers": args.layers,
                       "projections": 7 * args.layers, "mode": args.mode,
                       "timed_per_step": {"tokens": n_tok, "layers": rep, "projections": 7 * rep},
                       "step_equivalents_timed": toks / 512 / args.layers},
            "timed_seconds": total, "tokens_layers_evaluated": toks,
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample,
                             "single_thread": {"value": v1, "unit": "tokens/s", "cores": 1,
                                               "sample": f"{n1} tokens x 7 projections x 1 layer ({d1:.1f} s)"},
                             "cores_source": "os.sched_getaffinity"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def huge_page_bytes(ptr: int):
    """(mapping bytes, bytes backed by transparent huge pages) of the process
    mapping that holds `ptr`, from /proc/self/smaps; (None, None) if unknown."""
    try:
        cur = None
        with open("/proc/self/smaps") as f:
            for line in f:
                head = line.split(" ", 1)[0]
                if "-" in head and ":" not in head:
                    a, b = (int(x, 16) for x in head.split("-"))
                    cur = [b - a, None] if a <= ptr < b else None
                elif cur is not None and line.startswith("AnonHugePages:"):
                    cur[1] = int(line.split()[1]) * 1024
                    return cur[0], cur[1]
    except (OSError, ValueError):
        pass
    return None, None


def traffic_from_profile():
    """Per-launch DRAM traffic from the committed ncu summary, if it was taken
    on the current kernel source; else None."""
    p = os.path.join(ROOT, "profiles", "salt_apply_kernel_traffic.json")
    src = os.path.join(ROOT, "paper_2608_03579_gb300", "csrc", "salt_apply.cu")
    if not os.path.exists(p):
        return None, None
    d = json.load(open(p))
    h = hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]
    if d.get("kernel_source_sha256_16") != h:
        return None, None
    return d.get("dram_bytes_per_algorithmic_byte"), d


class DeviceErrors:
    """Reads (and clears) the library's device error word at checkpoints of a
    run.  A bounded in-kernel wait that gave up (SALT_DEVERR_TIMEOUT) or an id
    the kernels rejected means the launches of that stretch did less than the
    claimed work, so any number measured over it is invalid."""

    def __init__(self, salt_mod, ctx):
        self.salt, self.ctx = salt_mod, ctx
        self.seen = {}

    def check(self, where: str, stream=None) -> int:
        flags = int(self.salt.salt_get_device_error(self.ctx, stream))
        if flags:
            self.seen[where] = flags
        return flags

    @property
    def valid(self) -> bool:
        return not self.seen

    def summary(self):
        return {"valid": self.valid, "device_error_flags": {k: hex(v) for k, v in self.seen.items()}}


def host_link_rates(salt_mod, torch, device: int, nbytes: int = 1 << 30) -> dict:
    """H2D and D2H copy rates (GB/s) of one large copy each, from and to
    huge-page page-locked host memory, timed alone with CUDA events."""
    hb = salt_mod.salt_host_alloc(nbytes)
    h = hb.tensor
    d = torch.empty(nbytes, dtype=torch.uint8, device=f"cuda:{device}")
    s = torch.cuda.Stream(device=device)
    out = {}
    for name, (dst, src) in (("h2d_gbs", (d, h)), ("d2h_gbs", (h, d))):
        with torch.cuda.stream(s):
            dst.copy_(src, non_blocking=True)  # warm
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            for _ in range(3):
                dst.copy_(src, non_blocking=True)
            e1.record(s)
        s.synchronize()
        out[name] = 3 * nbytes / (e0.elapsed_time(e1) / 1000.0) / 1e9
    del d
    hb.close()
    return out


def step_e2e(args, st, pg, local, world, derr) -> dict:
    """Whole steps on host activations: swaps, the segment build, then every
    grouped apply through salt_lora_apply_host (copies in and out owned and
    overlapped by the library); the step ends when the last y is back in
    host memory."""
    import torch
    salt = st.salt
    hb_x = salt.salt_host_alloc(st.x_elems * 2 + 4096)
    hb_y = salt.salt_host_alloc(st.y_elems * 2 + 4096)
    xh = hb_x.tensor[:st.x_elems * 2].view(torch.bfloat16)
    yh = hb_y.tensor[:st.y_elems * 2].view(torch.bfloat16)
    xh.copy_(st.x_all)
    yh.zero_()
    xs = [xh[st.x_off[l]:st.x_off[l] + st.T * st.w.layers[l][1]] for l in range(st.L)]
    ys = [yh[st.y_off[l]:st.y_off[l] + st.T * st.w.layers[l][2]] for l in range(st.L)]
    largest = max(sum(st.T * (st.w.layers[l][1] + st.w.layers[l][2]) * 2 + 512 for l in grp) for grp in st.groups)
    pipe = salt.salt_host_pipe_create(st.runner.ctx, 3, largest)

    def one(s):
        st.swap(s)
        st.build(s)
        for grp in st.groups:
            salt.salt_lora_apply_host(pipe, st.runner.seg, grp, [xs[l] for l in grp], [ys[l] for l in grp], st.comp)
        salt.salt_host_pipe_wait(pipe, st.comp)

    base = args.warmup + args.steps + 16
    one(base)
    st.join_side()
    torch.cuda.synchronize(local)
    n_e2e = max(3, min(args.steps, 10))
    barrier(pg, local)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(st.comp)
    for s in range(n_e2e):
        one(base + 1 + s)
    st.join_side()
    e1.record(st.comp)
    torch.cuda.synchronize(local)
    derr.check("e2e")
    e2e_ms = max_over_ranks(pg, e0.elapsed_time(e1), local) / n_e2e
    pipe.close()
    rates = host_link_rates(salt, torch, local)
    hb_x.close()
    hb_y.close()
    h2d_act = st.x_elems * 2 + st.y_elems * 2
    h2d = h2d_act + 2 * st.T * 4 + st.wl_mod.C4_REGION * st.blob_bytes
    d2h = st.y_elems * 2
    return {"value": world * st.T / (e2e_ms / 1000.0), "unit": "tokens/s", "ms_per_step": e2e_ms,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "api": "salt_lora_apply_host (library-owned copies, 3 staging areas, H2D and D2H streams)",
            "host_link": rates,
            "bound_ms_at_host_link": {"h2d": 1000.0 * h2d / (rates["h2d_gbs"] * 1e9),
                                      "d2h": 1000.0 * d2h / (rates["d2h_gbs"] * 1e9)}}


def run_salt(args, rank, world, local, pg):
    import torch
    import __graft_entry__
    __graft_entry__.build()
    torch.cuda.set_device(local)
    peaks, peak_kind = load_peaks()
    st = Step(args, local)
    derr = DeviceErrors(st.salt, st.runner.ctx)
    ctx_info = st.salt.salt_ctx_get_info(st.runner.ctx)
    st.capture()
    per_group_bytes = st.apply_bytes()
    step_apply_bytes = float(per_group_bytes.sum())
    n_launch = len(st.groups)

    # warm-up
    for s in range(args.warmup):
        st.step(s)
    st.join_side()
    torch.cuda.synchronize(local)
    derr.check("warmup")

    # timed region: K whole steps
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        if not uuid.startswith("GPU-"):
            uuid = "GPU-" + uuid
    except Exception:
        uuid = None
    sampler = ClockSampler(uuid, f"{args.clocks_csv}.rank{rank}" if args.clocks_csv else None)
    barrier(pg, local)
    torch.cuda.synchronize(local)
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    # Only the two events that bound the timed region: an event pair recorded
    # around every step's graph launch was measured to delay the side-stream
    # swaps and lengthen the step by up to 2x.
    with sampler:
        time.sleep(0.3)
        t_start.record(st.comp)
        for s in range(args.warmup, args.warmup + args.steps):
            st.step(s)
        st.join_side()
        t_end.record(st.comp)
        torch.cuda.synchronize(local)
        time.sleep(0.2)
    ms_total = t_start.elapsed_time(t_end)
    derr.check("timed")
    barrier(pg, local)
    # per-launch durations of the apply kernel: a pass of whole steps right
    # after the timed region (swaps still overlapping), with an event pair on
    # the launching stream around every apply launch
    n_prof = 3
    launch_ms = np.zeros(len(st.groups))
    for s in range(n_prof):
        evs = st.step(args.warmup + args.steps + s, timing=True)
        st.join_side()
        torch.cuda.synchronize(local)
        launch_ms += np.array([a.elapsed_time(b) for (a, b) in evs])
    derr.check("per_launch_timing")
    kernel_ms = list(launch_ms / n_prof)
    kinds = ["qkv", "o", "gate_up", "down"]
    per_kind = {}
    for i, k in enumerate(kinds):
        msk = sum(kernel_ms[i::4])
        per_kind[k] = {"us_per_launch": 1000.0 * msk / (len(kernel_ms) // 4),
                       "GB/s": float(per_group_bytes[i::4].sum() / (msk / 1000.0) / 1e9)}
    # The applies alone: the step's graph of 128 grouped applies replayed
    # back to back (same tables as the last timed step, no swaps), an event
    # pair on the launching stream around each replay.  Its mean over the
    # 128 launches is the apply kernel's duration used for the roofline.
    apply_only_ms = None
    n_rep = 10
    reps = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n_rep)]
    for a, b in reps:
        a.record(st.comp)
        st.applies()
        b.record(st.comp)
    torch.cuda.synchronize(local)
    apply_only_ms = float(np.mean([a.elapsed_time(b) for (a, b) in reps]))
    derr.check("apply_only_replays")
    apply_ms_timed = apply_only_ms
    ms_total = max_over_ranks(pg, ms_total, local)
    ms_per_step = ms_total / args.steps
    value = world * st.T * args.steps / (ms_total / 1000.0)
    clocks = sampler.summary()

    # kernel roofline (the apply kernel dominates the step)
    roof = None
    if apply_ms_timed > 0:
        # the dominant kernel: one salt_apply_kernel launch per grouped apply,
        # its average duration from the graph replays above
        achieved = step_apply_bytes / (apply_ms_timed / 1000.0) / 1e9
        ratio, prof = traffic_from_profile()
        roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / peaks["hbm_gbs"],
                "traffic": (ratio * step_apply_bytes / n_launch) if ratio else None,
                "kernel": "salt_apply_kernel (one launch per grouped apply)",
                "launches_per_step": n_launch,
                "algorithmic_bytes_per_launch": step_apply_bytes / n_launch,
                "avg_launch_us": 1000.0 * apply_ms_timed / n_launch,
                "avg_launch_us_eager_pass": 1000.0 * sum(kernel_ms) / n_launch,
                "peak_kind": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"
                if peak_kind == "measured" else "fallback 6.8 TB/s"}

    # e2e: the step on host activations through the library's host pipe
    # (salt_lora_apply_host): per grouped apply, its x and y_in are copied in,
    # applied and y is copied out by the library, the copies of neighbouring
    # groups overlapping the applies on two copy streams
    e2e = None
    if not args.no_e2e:
        e2e = step_e2e(args, st, pg, local, world, derr)

    # swap-only and apply-only reference timings (context for the step time)
    swap_ms = None
    try:
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize(local)
        a.record(st.side)
        for s in range(4):
            st.swap(args.warmup + s)
        b.record(st.side)
        torch.cuda.synchronize(local)
        swap_ms = a.elapsed_time(b) / 4
    except Exception:
        swap_ms = None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline_line(args.mode, args.layers, args.cpu_seconds)

    derr.check("end")
    st.close()
    valid = max_over_ranks(pg, 0.0 if derr.valid else 1.0, local) == 0.0
    if rank == 0:
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": (WORKLOAD if args.mode == "salt" else WORKLOAD + "_rank16_lora")
                           + ("_gamma_bins" if args.gamma_bins else ""),
                           "tokens_per_step": st.T, "layers": args.layers, "projections": st.L,
                           "domains": 8, "centroid_rank": 0 if args.mode == "rank16" else 64,
                           "residual_rank": 16 if args.mode == "rank16" else 2, "slots": 512,
                           "swaps_per_step": 64, "swap_bytes_per_step": 64 * st.blob_bytes,
                           "apply_bytes_per_step": step_apply_bytes,
                           "l2": "inputs larger than L2 (the step streams > 8 GB; L2 is 126 MB)",
                           "parallelism": f"replicas x{world}", "launch": "CUDA graph of 128 grouped applies"},
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": args.steps * (n_launch + 1),
                "clocks": {k: clocks[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
                "swap_ms_per_step_alone": swap_ms, "apply_only_ms_per_step": apply_only_ms,
                "swap_host_memory": dict(zip(("bytes", "huge_page_bytes"), st.host_huge)),
                "apply_kernel_by_group": per_kind,
                "apply_launch_shape": {k: ctx_info[k] for k in ("apply_ctas", "k_splits_max", "apply_smem_bytes",
                                                                  "block_tokens", "block_users")},
                **derr.summary(), "valid": valid}
        print(json.dumps(line), flush=True)
    if not valid:
        print("device error flags were raised during the run; its numbers are invalid: "
              + json.dumps(derr.summary()), file=sys.stderr)
        raise SystemExit(3)


# ----------------------------------------------------------------------------- the other serving configurations
CONFIG_INFO = {
    1: ("llama3b_decode_qkv", 28, "Llama-3.2-3B q/k/v decode, 64 tokens, 4 domains rank 16, 64 users rank 2; "
        "one grouped q/k/v launch per layer, 28 layers (each its own factors and activations) replayed from "
        "one CUDA graph"),
    2: ("llama3b_prefill_mlp", 1, "Llama-3.2-3B MLP prefill, 8192 tokens in user segments of 128-1024, "
        "4 domains rank 32, residual ranks 1 and 2; gate/up grouped, then down"),
    3: ("llama8b_layer_decode", 8, "Llama-3.1-8B one layer (q, k, v, o, gate, up, down), 256 decode tokens, "
        "8 domains rank 64, 256 users rank 2 drawn Zipf(1.1); 4 grouped launches per layer, 8 copies of the "
        "layer (each its own factors and activations) replayed from one CUDA graph"),
}


def config_workload(wl, cfg: int):
    """The configuration's workload with its projections repeated over R
    layers, each with its own factors and activations (so a replay streams
    from HBM, not L2), and the groups of every copy."""
    w0 = wl.CONFIGS[cfg]()
    name, R, _ = CONFIG_INFO[cfg]
    L0 = len(w0.layers)
    layers = [(f"c{k}.{n}", a, b) for k in range(R) for (n, a, b) in w0.layers]
    groups = [[k * L0 + i for i in g] for k in range(R) for g in w0.group]
    w = wl.Workload(name, w0.seed, layers, w0.n_domains, list(w0.rc), w0.n_slots, list(w0.r_u),
                    dom_ids=w0.dom_ids, slot_ids=w0.slot_ids, group=groups)
    return w0, w, R


def config_cpu_baseline(w0, seconds: float) -> dict:
    """The fp64 oracle on a bounded sample of the configuration's tokens over
    all its projections, single-threaded and on every core (tokens split
    over host threads); tokens/s = tokens evaluated through every projection
    of the configuration / seconds."""
    import oracle
    oracle.build()
    cores = host_cores()
    tables = []
    used = set(int(u) for u in w0.slot_ids if u >= 0)
    for l in range(len(w0.layers)):
        cents = [(w0.centroid_At(d, l), w0.centroid_B(d, l), w0.s_c[d]) for d in range(w0.n_domains)]
        res = [((w0.residual_At(u, l), w0.residual_B(u, l), w0.s_u[u]) if u in used else None)
               for u in range(w0.n_slots)]
        tables.append((w0.x(l), w0.y_in(l), cents, res))

    def run(rows, threads, reps=1):
        parts = [q for q in np.array_split(rows, max(1, min(threads, len(rows)))) if len(q)]

        def work(part):
            for _ in range(reps):
                for (x, y, cents, res) in tables:
                    oracle.apply(x, y, w0.dom_ids, w0.slot_ids, cents, res, rows=part)

        t0 = time.perf_counter()
        ts = [threading.Thread(target=work, args=(q,)) for q in parts]
        for t in ts:
            t.start()
        for t in ts:
            t.join()
        return time.perf_counter() - t0

    out = {}
    for th in sorted({1, cores}):
        probe = np.linspace(0, w0.T - 1, min(w0.T, 2 * th)).round().astype(np.int64)
        dt = run(probe, th)
        want = (seconds / 2) / max(dt / len(probe), 1e-9)
        n = int(max(th, min(w0.T, want)))
        reps = max(1, int(round(want / w0.T))) if want > w0.T else 1
        rows = np.unique(np.linspace(0, w0.T - 1, n).round().astype(np.int64))
        dt = run(rows, th, reps)
        out[th] = (len(rows) * reps / dt, len(rows), reps, dt)
    (v1, n1, r1, d1), (vn, nn, rn, dn) = out[1], out[cores]
    return {"value": vn, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "sample": f"{nn} of the {w0.T} tokens through all {len(w0.layers)} projections, x{rn}, on {cores} "
                      f"threads ({dn:.1f} s); fp64 C oracle, tokens split over threads",
            "single_thread": {"value": v1, "unit": "tokens/s", "cores": 1,
                              "sample": f"{n1} tokens through all {len(w0.layers)} projections, x{r1} ({d1:.1f} s)"},
            "cores_source": "os.sched_getaffinity"}


def run_config(args, rank, world, local, pg):
    """One JSON line for serving configuration 1, 2 or 3: the configuration's
    grouped applies (R copies of its projections, so that every replay
    streams from HBM) captured in one CUDA graph and replayed; the roofline
    of the apply kernel; the oracle baseline; e2e through salt_lora_apply_host."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_03579_gb300 import salt
    from paper_2608_03579_gb300 import workloads as wl
    from paper_2608_03579_gb300.runner import SaltRunner
    torch.cuda.set_device(local)
    peaks, peak_kind = load_peaks()
    cfg = args.config
    w0, w, R = config_workload(wl, cfg)
    T, L0 = w.T, len(w0.layers)
    runner = SaltRunner(w, device=local, max_tokens=T)
    derr = DeviceErrors(salt, runner.ctx)
    runner.pin_centroids()
    runner.load_slots()
    comp = torch.cuda.Stream(device=local)
    runner.build(stream=comp)
    xs, ys = [], []
    gen = torch.Generator(device=f"cuda:{local}")
    gen.manual_seed(cfg)
    for l in range(len(w.layers)):
        din, dout = w.layers[l][1], w.layers[l][2]
        xs.append(torch.randn(T, din, generator=gen, device=f"cuda:{local}").to(torch.bfloat16))
        ys.append(torch.zeros(T, dout, dtype=torch.bfloat16, device=f"cuda:{local}"))

    def applies():
        for grp in w.group:
            salt.salt_lora_apply_grouped(runner.ctx, runner.seg, grp, [xs[l] for l in grp], [ys[l] for l in grp], comp)

    with torch.cuda.stream(comp):
        applies()
    torch.cuda.synchronize(local)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=comp):
        applies()
    for _ in range(args.warmup):
        with torch.cuda.stream(comp):
            graph.replay()
    torch.cuda.synchronize(local)
    derr.check("warmup")
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    sampler = ClockSampler(uuid, f"{args.clocks_csv}.rank{rank}" if args.clocks_csv else None)
    barrier(pg, local)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with sampler:
        time.sleep(0.2)
        e0.record(comp)
        for _ in range(args.steps):
            with torch.cuda.stream(comp):
                graph.replay()
        e1.record(comp)
        torch.cuda.synchronize(local)
    derr.check("timed")
    ms_replay = max_over_ranks(pg, e0.elapsed_time(e1), local) / args.steps
    ms_pass = ms_replay / R  # one pass of the configuration's projections
    value = world * T / (ms_pass / 1000.0)
    alg = float(sum(w0.algorithmic_bytes(l) for l in range(L0)))
    flops = float(sum(w0.algorithmic_flops(l) for l in range(L0)))
    launches_per_pass = len(w0.group)
    achieved = alg / (ms_pass / 1000.0) / 1e9
    roof = {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": achieved / peaks["hbm_gbs"], "traffic": None,
            "kernel": "salt_apply_kernel (one launch per grouped apply)",
            "launches_per_pass": launches_per_pass, "algorithmic_bytes_per_pass": alg,
            "avg_launch_us": 1000.0 * ms_pass / launches_per_pass,
            "peak_kind": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
            "tensor": {"achieved_tflops": flops / (ms_pass / 1000.0) / 1e12,
                       "peak_tflops": peaks.get("bf16_tflops"),
                       "frac": flops / (ms_pass / 1000.0) / 1e12 / peaks["bf16_tflops"] if peaks.get("bf16_tflops") else None,
                       "note": "algorithmic flops 2 (rc + r)(d_in + d_out) per token; the tensor cores run the "
                               "padded stacks, more than this"}}
    # e2e: the same pass on host activations
    e2e = None
    if not args.no_e2e:
        shapes = []
        for l in range(len(w.layers)):
            shapes += [T * w.layers[l][1], T * w.layers[l][2]]
        offs = np.cumsum([0] + [(n * 2 + 255) // 256 * 256 for n in shapes])
        hb = salt.salt_host_alloc(int(offs[-1]))
        views = [hb.tensor[int(o):int(o) + n * 2].view(torch.bfloat16) for o, n in zip(offs, shapes)]
        xh, yh = views[0::2], views[1::2]
        for l in range(len(w.layers)):
            xh[l].copy_(xs[l].view(-1))
            yh[l].zero_()
        largest = max(sum(T * (w.layers[l][1] + w.layers[l][2]) * 2 + 512 for l in grp) for grp in w.group)
        pipe = salt.salt_host_pipe_create(runner.ctx, 3, largest)

        def host_pass():
            for grp in w.group:
                salt.salt_lora_apply_host(pipe, runner.seg, grp, [xh[l] for l in grp], [yh[l] for l in grp], comp)
            salt.salt_host_pipe_wait(pipe, comp)

        host_pass()
        torch.cuda.synchronize(local)
        n_e2e = max(2, min(args.steps, 5))
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(comp)
        for _ in range(n_e2e):
            host_pass()
        b.record(comp)
        torch.cuda.synchronize(local)
        derr.check("e2e")
        e2e_ms_pass = max_over_ranks(pg, a.elapsed_time(b), local) / n_e2e / R
        pipe.close()
        hb.close()
        rates = host_link_rates(salt, torch, local)
        h2d = sum(T * (w0.layers[l][1] + w0.layers[l][2]) * 2 for l in range(L0))
        d2h = sum(T * w0.layers[l][2] * 2 for l in range(L0))
        e2e = {"value": world * T / (e2e_ms_pass / 1000.0), "unit": "tokens/s", "ms_per_pass": e2e_ms_pass,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "api": "salt_lora_apply_host", "host_link": rates,
               "bound_ms_at_host_link": {"h2d": 1000.0 * h2d / (rates["h2d_gbs"] * 1e9),
                                         "d2h": 1000.0 * d2h / (rates["d2h_gbs"] * 1e9)}}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = config_cpu_baseline(w0, args.cpu_seconds)
    derr.check("end")
    clocks = sampler.summary()
    valid = max_over_ranks(pg, 0.0 if derr.valid else 1.0, local) == 0.0
    runner.close()
    if rank == 0:
        name, _, desc = CONFIG_INFO[cfg]
        line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_replay, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": name, "config_index": cfg, "description": desc, "tokens": T,
                           "projections_per_pass": L0, "copies_per_replay": R,
                           "step": f"one CUDA-graph replay = {R} pass(es) of the configuration's projections",
                           "algorithmic_bytes_per_pass": alg,
                           "l2": "inputs larger than L2: each replay streams R distinct copies"
                                 if R > 1 else "inputs larger than L2 (882 MB per pass)",
                           "parallelism": f"replicas x{world}"},
                "roofline": roof, "cpu_baseline": cpu, "e2e": e2e,
                "gpu_launches": args.steps * R * launches_per_pass,
                "clocks": {k: clocks[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
                **derr.summary(), "valid": valid}
        print(json.dumps(line), flush=True)
    if not valid:
        raise SystemExit(3)


# ----------------------------------------------------------------------------- other rows of the path
def run_row(args, rank, world, local, pg):
    """One JSON line for the centroid fold or the alignment regulariser over
    the 224 adapted matrices of Llama-3.1-8B (32 layers x q, k, v, o, gate,
    up, down), timed with CUDA events on the launching stream."""
    import torch
    import __graft_entry__
    __graft_entry__.build()
    from paper_2608_03579_gb300 import salt
    from paper_2608_03579_gb300 import workloads as wl
    torch.cuda.set_device(local)
    peaks, peak_kind = load_peaks()
    shapes = [(din, dout) for _ in range(args.layers) for (_, din, dout) in wl.LLAMA8B_LAYER]
    n = len(shapes)
    stream = torch.cuda.Stream(device=local)
    gen = torch.Generator(device=f"cuda:{local}")
    gen.manual_seed(4)

    def randn(*shape, std=1.0):
        return (torch.randn(*shape, generator=gen, device=f"cuda:{local}") * std).to(torch.bfloat16)

    rc = 64
    runner = None
    flops = None
    if args.row == "base":
        # y = x W_base + the SALT delta for the 7 projections of one Llama-3.1-8B
        # layer, the 512-token decode batch of the step (8 rank-64 centroids,
        # rank-2 residuals drawn Zipf(1.1)); W_base as a linear layer stores it
        from paper_2608_03579_gb300.runner import SaltRunner
        w = wl.config4(seed=4, step=1, n_layers=1)
        runner = SaltRunner(w, device=local, max_tokens=w.T)
        runner.pin_centroids()
        runner.load_slots()
        runner.build(stream=stream)
        torch.cuda.synchronize(local)
        shapes = [(din, dout) for (_, din, dout) in w.layers]
        n = len(shapes)
        T = w.T
        W = [randn(b, a, std=a ** -0.5) for (a, b) in shapes]
        X = [randn(T, a) for (a, _) in shapes]
        Y = [torch.empty(T, b, dtype=torch.bfloat16, device=f"cuda:{local}") for (_, b) in shapes]
        ctx = None
        flops = float(sum(2.0 * T * a * b for a, b in shapes) + sum(w.algorithmic_flops(l) for l in range(n)))
        alg = float(sum(a * b * 2 + T * a * 2 + T * b * 2 for a, b in shapes)
                    + sum(w.algorithmic_bytes(l) - T * (a * 2 + b * 4) for l, (a, b) in enumerate(shapes)))

        def one(k):
            for l in range(n):
                salt.salt_lora_apply_with_base(runner.ctx, runner.seg, l, X[l], W[l], salt.SALT_W_OUT_IN, Y[l], stream)

        def step_pair():
            one(0)
            one(1)
        metric, unit, what = ("base GEMM fused with the SALT delta, TFLOP/s (y = x W_base + delta, one layer)",
                              "TFLOP/s", "llama8b_layer_base_plus_delta_512tok")
    elif args.row == "fold":
        d_in = [a for a, _ in shapes]
        d_out = [b for _, b in shapes]
        ctx = salt.salt_ctx_create(d_in, d_out, 1, rc, 1, 1, 16, local)
        A = np.concatenate([wl.normal_bf16(4, wl.stream_id(wl.K_CENT_A, 0, l), rc * a, 1 / np.sqrt(a))
                            for l, (a, _) in enumerate(shapes)])
        B = np.concatenate([wl.normal_bf16(4, wl.stream_id(wl.K_CENT_B, 0, l), rc * b, 1 / np.sqrt(rc))
                            for l, (_, b) in enumerate(shapes)])
        salt.salt_centroid_pin(ctx, 0, rc, A, B, 1.0)
        # base weights as a linear layer stores them, [d_out][d_in]
        W = [randn(b, a, std=0.02) for (a, b) in shapes]
        w_bytes = sum(a * b * 2 for a, b in shapes)
        alg = 2 * w_bytes + sum(rc * (a + b) * 2 for a, b in shapes)

        # one fold plan over all 224 weights: one launch per pass
        plan = salt.salt_fold_plan_create(ctx, 0, list(range(n)), W, salt.SALT_W_OUT_IN)

        def one(k):
            salt.salt_fold_plan_run(plan, 0.8 if k % 2 == 0 else -0.8, stream)
        # a step = +gamma then -gamma over every matrix, captured once
        def step_pair():
            one(0)
            one(1)
        metric, unit, what = "centroid fold GB/s (W += gamma s_c A_c B_c over every adapted weight)", "GB/s", \
            "llama8b_32layer_centroid_fold_rank64"
    else:
        r = 16
        keep, pairs = [], []
        for (a, b) in shapes:
            t = (randn(r, a, std=a ** -0.5), randn(r, b, std=r ** -0.5), randn(rc, a, std=a ** -0.5),
                 randn(rc, b, std=rc ** -0.5))
            keep.append(t)
            pairs.append(dict(At=t[0], B=t[1], At_c=t[2], B_c=t[3], r=r, rc=rc, d_in=a, d_out=b, s=1.0, s_c=1.0))
        loss = torch.empty(n, device=f"cuda:{local}")
        alg = sum((r + rc) * (a + b) * 2 for a, b in shapes)
        ctx = None
        arr = salt.salt_align_pairs(pairs)

        def one(k):
            salt.salt_align_loss(arr, 1e-8, loss, None, stream)

        def step_pair():
            one(0)
            one(1)
        metric, unit, what = "alignment regulariser GB/s (Eq. 2, factored, every adapted weight)", "GB/s", \
            "llama8b_32layer_align_rank16_vs_rank64"
    for k in range(args.warmup):
        one(k)
    torch.cuda.synchronize(local)
    # the launches of two steps captured in one CUDA graph (the host-side
    # marshalling of 224 calls would otherwise pace the GPU)
    graph = None
    try:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            step_pair()
        graph = g
    except Exception as e:
        print(f"graph capture failed ({e}); timing eager calls", file=sys.stderr)
        torch.cuda.synchronize(local)
    if graph is not None:
        for _ in range(2):
            with torch.cuda.stream(stream):
                graph.replay()
        torch.cuda.synchronize(local)
    n_pairs_timed = (args.steps + 1) // 2
    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(local).uuid)
        uuid = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
    except Exception:
        pass
    sampler = ClockSampler(uuid, f"{args.clocks_csv}.rank{rank}" if args.clocks_csv else None)
    barrier(pg, local)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    with sampler:
        time.sleep(0.2)
        e0.record(stream)
        if graph is not None:
            with torch.cuda.stream(stream):
                for k in range(n_pairs_timed):
                    graph.replay()
        else:
            for k in range(2 * n_pairs_timed):
                one(args.warmup + k)
        e1.record(stream)
        torch.cuda.synchronize(local)
    steps_done = 2 * n_pairs_timed
    ms = max_over_ranks(pg, e0.elapsed_time(e1), local) / steps_done
    achieved = alg / (ms / 1000.0) / 1e9
    clocks = sampler.summary()
    flags = salt.salt_get_device_error(runner.ctx if runner is not None else ctx, None) if (runner or ctx) else 0
    if args.row == "fold":
        salt.salt_fold_plan_destroy(plan)
    if ctx is not None:
        salt.salt_ctx_destroy(ctx)
    if runner is not None:
        runner.close()
    if rank == 0 and args.row == "base":
        tflops = flops / (ms / 1000.0) / 1e12
        peak_t = peaks.get("bf16_tflops", PEAKS_FALLBACK["bf16_tflops"])
        print(json.dumps({
            "metric": metric, "value": world * tflops, "unit": unit, "n_gpus": world, "steps": steps_done,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": what, "tokens": T, "projections": n, "w_layout": "[d_out][d_in]",
                       "flops_per_step": flops, "algorithmic_bytes_per_step": alg,
                       "l2": "inputs larger than L2 (218 MB of base weights per layer)",
                       "launch": "CUDA graph of two steps (per projection: a shrink-only apply, then the fused GEMM)"},
            "roofline": {"bound": "tensor", "achieved": tflops, "peak": peak_t, "unit": "TFLOP/s",
                         "frac": tflops / peak_t, "traffic": None,
                         "hbm": {"achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                                 "frac": achieved / peaks["hbm_gbs"]}},
            "gpu_launches": steps_done * 2 * n, "valid": flags == 0,
            "clocks": {k: clocks[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")}}), flush=True)
    elif rank == 0:
        launches = 1 if args.row == "fold" else (n + 255) // 256
        print(json.dumps({
            "metric": metric, "value": world * achieved, "unit": unit, "n_gpus": world, "steps": steps_done,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": what, "matrices": n, "algorithmic_bytes_per_step": alg,
                       "l2": "inputs larger than L2", "launch": ("CUDA graph of two steps" if graph is not None
                       else "eager calls") + ("; one fold-plan launch per step" if args.row == "fold" else "")},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": achieved / peaks["hbm_gbs"], "traffic": None},
            "gpu_launches": steps_done * launches, **({"valid": flags == 0} if args.row == "fold" else {}),
            "clocks": {k: clocks[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")}}), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        # the oracle arm runs on rank 0's host cores alone; no process group
        run_reference(args, int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), None)
        return
    rank, world, local, pg = dist_setup(args)
    try:
        if args.row != "step":
            run_row(args, rank, world, local, pg)
        elif args.config != 4:
            run_config(args, rank, world, local, pg)
        else:
            run_salt(args, rank, world, local, pg)
    finally:
        if pg is not None:
            pg.destroy_process_group()


if __name__ == "__main__":
    main()
