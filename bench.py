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
    ap.add_argument("--row", default="step", choices=["step", "fold", "align"])
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
        for i in range(self.wl_mod.C4_REGION):
            self.salt.salt_residual_load(self.runner.ctx, region + i, hs[i], self.side)

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

    # e2e: host buffers, copies inside the timed region
    e2e = None
    if not args.no_e2e:
        # host activations in huge-page page-locked memory (salt_host_alloc):
        # ordinary pinned pages stall the copy engine under sustained transfers
        hb = [st.salt.salt_host_alloc(n * 2) for n in (st.x_elems, st.y_elems, st.y_elems)]
        x_host, y_host, y_out = (h.tensor.view(torch.bfloat16) for h in hb)
        x_host.copy_(st.x_all)
        y_host.zero_()
        torch.cuda.synchronize(local)
        n_e2e = max(3, min(args.steps, 10))
        barrier(pg, local)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(st.comp)
        for s in range(n_e2e):
            with torch.cuda.stream(st.comp):
                st.x_all.copy_(x_host, non_blocking=True)
                st.y_all.copy_(y_host, non_blocking=True)
            st.step(args.warmup + args.steps + s)
            with torch.cuda.stream(st.comp):
                y_out.copy_(st.y_all, non_blocking=True)
        st.join_side()
        e1.record(st.comp)
        torch.cuda.synchronize(local)
        derr.check("e2e")
        e2e_ms = max_over_ranks(pg, e0.elapsed_time(e1), local) / n_e2e
        h2d = st.x_elems * 2 + st.y_elems * 2 + 2 * st.T * 4 + st.wl_mod.C4_REGION * st.blob_bytes
        e2e = {"value": world * st.T / (e2e_ms / 1000.0), "unit": "tokens/s", "ms_per_step": e2e_ms,
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(st.y_elems * 2)}
        x_host = y_host = y_out = None
        for h in hb:
            h.close()

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
                "apply_kernel_by_group": per_kind,
                "apply_launch_shape": {k: ctx_info[k] for k in ("apply_ctas", "k_splits_max", "apply_smem_bytes",
                                                                  "block_tokens", "block_users")},
                **derr.summary(), "valid": valid}
        print(json.dumps(line), flush=True)
    if not valid:
        print("device error flags were raised during the run; its numbers are invalid: "
              + json.dumps(derr.summary()), file=sys.stderr)
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
    if args.row == "fold":
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

        def one(k):
            g = 0.8 if k % 2 == 0 else -0.8
            for l in range(n):
                salt.salt_centroid_fold(ctx, 0, l, g, W[l], salt.SALT_W_OUT_IN, stream)
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
    if ctx is not None:
        salt.salt_ctx_destroy(ctx)
    if rank == 0:
        launches = n if args.row == "fold" else 2 * ((n + 255) // 256)
        print(json.dumps({
            "metric": metric, "value": world * achieved, "unit": unit, "n_gpus": world, "steps": steps_done,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": what, "matrices": n, "algorithmic_bytes_per_step": alg,
                       "l2": "inputs larger than L2", "launch": "CUDA graph of two steps" if graph is not None
                       else "eager calls"},
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                         "frac": achieved / peaks["hbm_gbs"], "traffic": None},
            "gpu_launches": steps_done * launches,
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
        else:
            run_salt(args, rank, world, local, pg)
    finally:
        if pg is not None:
            pg.destroy_process_group()


if __name__ == "__main__":
    main()
