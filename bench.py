#!/usr/bin/env python3
"""Benchmark of the PPD verification step (tree attention over every layer,
node argmax, acceptance, KV compaction) through libppd's C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl reference]

Prints one JSON line.  The headline workload is the Vicuna-7B-shaped cache
(32 layers, 32 heads x 128, bf16 K/V, batch 1, prefix 2048, 64-token tree,
vocab 32000).  Inputs are seeded synthetic tensors resident in HBM.  When a
step's inputs are at least four times the 129 MB L2 (every Vicuna-shaped
workload: 1.17 GB per step at Vicuna-7B), steps run back to back and no step
can find the previous one's data in L2; smaller workloads flush L2 (a 256 MiB
write) before every timed step, outside the step's events.

On one GPU the default run also times, each with its own K steps, the other
workloads of the paper's evaluation models (MobileLlama-, Vicuna-13B-shaped,
and the batch-8 / prefix-16384 tree-size sweep) under "workloads", the
attention as a model calls it (one call per layer) under
"per_layer_attention", and the step latency against the tree size (the
hardware half of the paper's hardware-aware tree size) under
"tree_size_profile", and the steps after the verification path: the step
with typical acceptance under "typical_step" and next-step candidate
generation under "next_tree" (on the headline trees, and on trees of four
ensemble chains with the chains' logits or probabilities averaged).  GPU
clocks are sampled from before the first warm-up step to after the last
timed loop; "clocks" summarises the samples taken inside timed loops.

Under torchrun (N > 1) each rank runs an independent replica of the headline
workload on its own GPU (weak scaling: the sequences of different ranks are
independent, no data-path collective); the step time is the maximum over
ranks.  `--impl reference` times the fp64 CPU oracle on the host cores
instead (rank 0 only), on whole steps of the same workload when they fit a
few minutes, else on a bounded sample of each step.
"""
from __future__ import annotations

import argparse
import datetime
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "verify steps/s and achieved HBM GB/s (frac of ~8 TB/s), Vicuna-7B shapes"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_FLUSH_BYTES = 256 << 20
TYPICAL = (0.7, 0.09, 0.3)   # temperature, epsilon, delta of --accept typical
L2_BYTES = 129 * 1000 * 1000
# the other workloads of the paper's evaluation models, timed after the headline one
EXTRA_WORKLOADS = ("mobilellama", "vicuna13b", "sweep_t16", "sweep_t32", "sweep_t64", "sweep_t128")
# tree sizes of the latency profile L_fp(n) (Vicuna-7B shapes)
PROFILE_SIZES = (16, 32, 48, 64, 96, 128, 192, 256, 384, 512)
# seconds of oracle work the reference arm may spend in total before it falls
# back from whole steps to a bounded sample of each step
REFERENCE_BUDGET_S = 180.0

# DRAM traffic of one launch of the roofline kernel (dram__bytes_read.sum +
# dram__bytes_write.sum), keyed by workload, with the hash of the attention
# sources it was taken on: a stale entry reports null.  The captures ran the
# attention alone (ppd_tree_attention, the roofline kernel whenever the step
# is more than one launch) at the same shapes with 19 layers (608 / 760 units:
# whole rounds of 152 CTAs) and are scaled to the full layer count, since the
# traffic grows with the units.  Writes still held in L2 when the kernel ends
# are not in the count, so this is the reads plus the part of the writes that
# reached DRAM during the launch.
MEASURED_TRAFFIC = {
    # 676,148,224 B at 19 layers (reads 667,937,280), x 32/19
    "vicuna7b": {"bytes_per_launch": 1_138_775_956, "src": "2d25b5ff49083324"},
    # 1,659,156,992 B at 19 layers (reads 1,650,976,000), x 40/19
    "vicuna13b": {"bytes_per_launch": 3_492_962_088, "src": "2d25b5ff49083324"},
    # 123,574,016 B, a fused-step launch at the full 24 layers (reads 119,720,448)
    "mobilellama": {"bytes_per_launch": 123_574_016, "src": "2d25b5ff49083324"},
}


def attention_source_hash() -> str:
    h = hashlib.sha256()
    for f in ("ppd_attention.cu", "ppd_attention_rows.cu", "ppd_attention_common.cuh",
              "ppd_device.cuh", "ppd_accept.cuh", "ppd_kernels.h", "ppd_api.cu"):
        with open(os.path.join(ROOT, "paper_2405_18628_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_peak_gbs():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ----------------------------------------------------------------------------- bytes

def packed(specs, device):
    """One uint8 buffer holding several tensors, each at a 256-byte aligned
    offset: specs {name: (shape, dtype)} -> (buffer, {name: view}).  Host
    buffers are pinned when a GPU is present."""
    import torch
    offs, off = {}, 0
    for k, (shape, dt) in specs.items():
        n = int(np.prod(shape)) * torch.empty((), dtype=dt).element_size()
        offs[k] = (off, n)
        off += (n + 255) // 256 * 256
    buf = torch.empty(off, dtype=torch.uint8, device=device,
                      pin_memory=(str(device) == "cpu" and torch.cuda.is_available()))
    views = {k: buf[o:o + n].view(specs[k][1]).view(specs[k][0]) for k, (o, n) in offs.items()}
    return buf, views


def attention_bytes(w) -> int:
    """Algorithmic bytes of one tree-attention launch over all L*B*H slices:
    per slice the bf16 K/V prefix (4*P*D), tree K/V (4*T*D), Q (2*T*D) and the
    fp32 output (4*T*D)."""
    per_unit = 4 * w.P * w.D + 4 * w.T * w.D + 2 * w.T * w.D + 4 * w.T * w.D
    return w.L * w.B * w.H * per_unit


def step_bytes(w, n_acc_total: int) -> int:
    """Algorithmic bytes of one verification step: attention, the fp32 logits,
    the compacted K/V rows written into the cache (bf16 K and V: 4*D bytes per
    layer, head and accepted node; the tree rows they copy are already counted
    in the attention's reads) and the small integer arrays (parent, candidate
    ids, argmax and path per node; prefix, accepted length, next token, new
    prefix, status per sequence)."""
    ints = 4 * w.B * w.T * 4 + 4 * w.B * 6
    return (attention_bytes(w) + 4 * w.B * w.T * w.V +
            4 * w.L * w.H * w.D * n_acc_total + ints)


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling every 50 ms into a file, with the sample timestamps;
    `summary(windows)` keeps the samples inside the given (start, end)
    datetime windows (the timed loops)."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self, wait_s: float = 5.0):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            return self
        t0 = time.perf_counter()
        while time.perf_counter() - t0 < wait_s and not self._rows():
            time.sleep(0.05)
        return self

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.proc = None

    @staticmethod
    def _num(x):
        try:
            return float(x)
        except ValueError:
            return None

    def _rows(self):
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) < 10 or self._num(parts[2]) is None:
                        continue
                    try:
                        ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f")
                    except ValueError:
                        continue
                    rows.append((ts, parts))
        except Exception:
            pass
        return rows

    def summary(self, windows):
        rows = self._rows()
        if self.path and os.path.exists(self.path):
            os.unlink(self.path)
        inside = [r for ts, r in rows if any(a <= ts <= b for a, b in windows)]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "samples_in_timed_loops": 0}
        use = inside if inside else [r for _, r in rows]
        pw = [self._num(r[4]) for r in use if self._num(r[4]) is not None]
        reasons = sorted({self.REASONS[k] for r in use for k in range(4)
                          if r[6 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(self._num(r[2]) for r in use),
                "sm_max_mhz": max(self._num(r[3]) for r in use),
                "power_w_max": max(pw) if pw else None,
                "reasons": reasons, "samples": len(rows),
                "samples_in_timed_loops": len(inside),
                "basis": ("samples inside the timed loops" if inside else
                          "every sample of the run (none fell inside a timed loop)")}


class Windows:
    """Wall-clock windows of the timed loops (for the clock summary)."""

    def __init__(self):
        self.spans = []

    def __enter__(self):
        self._t0 = datetime.datetime.now()
        return self

    def __exit__(self, *exc):
        self.spans.append((self._t0, datetime.datetime.now()))


# ----------------------------------------------------------------------------- CPU oracle

def oracle_step_seconds(w, host, s, units, n_threads: int) -> float:
    """One fp64 oracle verification step on a sample of the workload, scaled to
    the whole step.  `host` holds the first few layers of Q/K/V on the host;
    attention runs on `units` of them (None: all), compaction on all of them,
    argmax and acceptance once, as in a full step.  Attention and compaction
    times are scaled by the fraction of the workload the sample covers (1 for
    a whole step)."""
    import oracle
    L_h = host["q"].shape[0]
    n_sample = len(units) if units is not None else L_h * w.B * w.H
    t0 = time.perf_counter()
    oracle.tree_attention(host["q"], host["k_cache"], host["v_cache"], host["k_tree"],
                          host["v_tree"], s.prefix_len, s.parent, units=units,
                          n_threads=n_threads)
    t_att = time.perf_counter() - t0
    t0 = time.perf_counter()
    am = oracle.node_argmax(s.logits)
    acc = oracle.accept_path(am, s.cand_tokens, s.parent, s.prefix_len, w.V, w.S_max)
    t_acc = time.perf_counter() - t0
    t0 = time.perf_counter()
    oracle.kv_compact(host["k_cache"], host["v_cache"], host["k_tree"], host["v_tree"],
                      acc["path"], acc["accept_len"], s.prefix_len)
    t_cmp = time.perf_counter() - t0
    return t_att * (w.L * w.B * w.H) / n_sample + t_acc + t_cmp * w.L / L_h


def one_thread_seconds(w, host, s) -> float:
    """The oracle step on one host thread: the attention of the first layer
    (all sequences and heads) scaled by L, argmax and acceptance in full."""
    one = {k: v[:1] for k, v in host.items()}
    return oracle_step_seconds(w, one, s, None, 1)


def cpu_baseline(w, t_dev, s, budget_s: float):
    """Oracle on the first `nl` layers, `nl` chosen from a one-layer calibration
    so the sample takes about `budget_s` seconds of host time."""
    n_threads = os.cpu_count() or 1
    one = {k: v[:1].cpu() for k, v in t_dev.items()}
    t0 = time.perf_counter()
    oracle_step_seconds(w, one, s, None, n_threads)
    t1 = time.perf_counter() - t0
    nl = max(1, min(w.L, int(budget_s / max(t1, 1e-6))))
    host = one if nl == 1 else {k: v[:nl].cpu() for k, v in t_dev.items()}
    sec = oracle_step_seconds(w, host, s, None, n_threads)
    return {"value": 1.0 / sec, "unit": "steps/s", "cores": n_threads, "kind": "oracle",
            "sample": (f"fp64 oracle verification step on all {w.L} layers (whole step)"
                       if nl == w.L else
                       f"fp64 oracle verification step on the first {nl} of {w.L} layers "
                       f"(all heads; attention and compaction time scaled by {w.L}/{nl}; "
                       f"full argmax and acceptance)")}


# ----------------------------------------------------------------------------- main

def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--config", default="vicuna7b")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--cpu-budget", type=float, default=12.0,
                    help="seconds of oracle work in the CPU baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-extras", action="store_true",
                    help="time the headline workload only (no other workloads, per-layer "
                         "attention or tree-size profile)")
    ap.add_argument("--accept", default="exact", choices=["exact", "typical"],
                    help="verification rule: exact matching, or typical acceptance at "
                         "temperature 0.7, epsilon 0.09, delta 0.3")
    ap.add_argument("--tree-sizes", default=None,
                    help="comma-separated tree sizes of the latency profile (the hardware "
                         "half of the paper's hardware-aware tree size); '' for none")
    ap.add_argument("--tau", default="",
                    help="JSON file {tree size: acceptance length}: also report "
                         "Speedup(n) = tau(n) / latency(n) and the best size")
    ap.add_argument("--next-tree", action="store_true",
                    help="also time next-step candidate generation (ppd_next_tree, 5 tree "
                         "states, 8 guesses per depth) after each step")
    ap.add_argument("--per-layer", action="store_true",
                    help="time the per-layer attention even when extras are off")
    ap.add_argument("--layers", type=int, default=0,
                    help="run the workload with this many layers (profiling captures)")
    ap.add_argument("--form", type=int, default=None, choices=[1, 2, 3],
                    help="force the fused step's form (1: argmax grid first; 2: argmax in the "
                         "side warps; 3: argmax in the softmax warps before their first tile)")
    ap.add_argument("--l2", default="auto", choices=["auto", "flush", "none"],
                    help="auto: flush L2 before each step unless the step's inputs exceed 4x L2")
    return ap.parse_args(argv)


def dist_setup(env=None):
    """(world size, rank, local rank) from the torchrun environment."""
    env = os.environ if env is None else env
    world = int(env.get("WORLD_SIZE", "1"))
    rank = int(env.get("RANK", "0"))
    local = int(env.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, dist=None, device="cpu") -> float:
    """The largest `value` over all ranks (the slowest rank's time)."""
    if dist is None:
        return value
    import torch
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def aggregate_rate(steps_per_rank: int, world: int, slowest_ms: float) -> float:
    """Whole-job steps/s: every rank's steps over the slowest rank's time."""
    return world * steps_per_rank / (slowest_ms / 1e3)


def resolve_workload(args):
    from paper_2405_18628_gb300 import workloads as W
    w = W.WORKLOADS[args.config]
    if args.layers:
        # fewer layers of the same shapes: small cases for profiler captures
        w = W.scaled(w, L=args.layers)
    return w


def flushes_l2(w, mode: str) -> bool:
    """Whether L2 is flushed before each timed step: always with "flush", never
    with "none", and with "auto" when a step's inputs are below 4x L2."""
    return mode == "flush" or (mode == "auto" and step_bytes(w, 0) < 4 * L2_BYTES)


def config_of(w, args, world: int) -> dict:
    """The `config` object of the JSON line (the same for both arms)."""
    footprint = step_bytes(w, 0)
    return {"workload": w.name + (f" ({w.L} layers)" if args.layers else ""),
            "layers": w.L, "batch": w.B, "heads": w.H, "head_dim": w.D, "prefix": w.P,
            "tree_tokens": w.T, "vocab": w.V, "S_max": w.S_max,
            "l2": ("flushed before every step (256 MiB write, outside the step events)"
                   if flushes_l2(w, args.l2) else
                   f"not flushed: inputs larger than L2 ({footprint / 1e6:.0f} MB "
                   f"streamed per step, L2 {L2_BYTES / 1e6:.0f} MB)"),
            "parallelism": f"replicas x{world}",
            "accept": ("exact matching" if args.accept == "exact" else
                       "typical acceptance (temperature %g, epsilon %g, delta %g)" % TYPICAL)}


def run_reference(args, w, world, rank):
    """The CPU oracle as the reference arm: whole verification steps of the
    workload (attention of every layer, argmax, acceptance, compaction of every
    layer) when W + K of them fit REFERENCE_BUDGET_S, else each step a bounded
    sample (a few attention slices of layer 0 scaled to all slices, the full
    argmax and acceptance, layer-0 compaction scaled to all layers).  Also a
    one-thread timing of the step (first layer scaled by L)."""
    if rank != 0:
        return
    from paper_2405_18628_gb300 import workloads as W

    s = W.make_step_inputs(w)
    n_threads = os.cpu_count() or 1
    host = W.make_tensors(w, device="cpu")
    t0 = time.perf_counter()
    oracle_step_seconds(w, host, s, None, n_threads)          # calibration (= warm-up 1)
    t_full = time.perf_counter() - t0
    whole = (args.warmup + args.steps) * t_full <= REFERENCE_BUDGET_S
    if whole:
        units = None
        sample = (f"whole steps: attention of all {w.L * w.B * w.H} slices, full argmax and "
                  f"acceptance, compaction of all {w.L} layers")
    else:
        per_step = max(0.01, REFERENCE_BUDGET_S / max(1, args.steps + args.warmup))
        n_all = w.L * w.B * w.H
        n_units = int(max(1, min(n_all, n_all * per_step / max(t_full, 1e-9))))
        units = list(range(n_units))
        sample = (f"{n_units} of {n_all} attention slices per step, scaled to all slices; "
                  f"full argmax and acceptance; compaction of all layers")
    for _ in range(max(0, args.warmup - 1)):
        oracle_step_seconds(w, host, s, units, n_threads)
    secs = [oracle_step_seconds(w, host, s, units, n_threads) for _ in range(args.steps)]
    sec_per_step = statistics.mean(secs)
    value = 1.0 / sec_per_step
    t1 = one_thread_seconds(w, host, s)
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sec_per_step * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": config_of(w, args, world),
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": n_threads, "kind": "oracle",
                         "sample": sample},
        "one_thread": {"value": 1.0 / t1, "unit": "steps/s", "cores": 1, "kind": "oracle",
                       "sample": f"attention of layer 0 (all heads) scaled by {w.L}; full argmax "
                                 f"and acceptance; compaction of layer 0 scaled by {w.L}"},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


class Step:
    """Device inputs and outputs of one workload and its step call."""

    def __init__(self, w, dev, seed, accept="exact"):
        import torch

        from paper_2405_18628_gb300 import ppd
        from paper_2405_18628_gb300 import workloads as W
        self.w, self.dev, self.accept = w, dev, accept
        self.s = W.make_step_inputs(w, seed=seed)
        self.t = W.make_tensors(w, device=dev, seed=seed)
        i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
        self.parent, self.cand, self.prefix = (i32(self.s.parent), i32(self.s.cand_tokens),
                                               i32(self.s.prefix_len))
        self.logits = torch.from_numpy(self.s.logits).to(dev)
        self.bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)

    def __call__(self, stream):
        from paper_2405_18628_gb300 import ppd
        t, b = self.t, self.bufs
        if self.accept == "typical":
            ppd.ppd_verify_step_typical(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                        self.prefix, self.parent, self.cand, self.logits, *TYPICAL,
                                        b.out, b.argmax, b.accept_len, b.path, b.next_token,
                                        b.new_prefix_len, b.dev_status, b.workspace, stream=stream)
        else:
            ppd.ppd_verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                self.prefix, self.parent, self.cand, self.logits, b.out, b.argmax,
                                b.accept_len, b.path, b.next_token, b.new_prefix_len,
                                b.dev_status, b.workspace, stream=stream)

    def check(self):
        status = self.bufs.dev_status.cpu().numpy()
        n_acc = int(self.bufs.accept_len.sum().item())
        if (status != 0).any() or n_acc < self.w.B:
            raise SystemExit(f"{self.w.name}: verification step reported device status "
                             f"{status.tolist()}")
        return n_acc


def head_start(stream):
    """A ~1 ms spin on `stream` ahead of a timed loop, outside its events: the
    host then queues the first calls before the GPU reaches them, so no step's
    events take in the host's launch latency (after the synchronize before a
    loop the stream is empty, and the first event would be timestamped at
    once)."""
    import torch
    with torch.cuda.stream(stream):
        torch.cuda._sleep(2_000_000)


def time_loop(fn, K, warmup, stream, flush, windows):
    """W untimed calls, then K calls each between CUDA events on `stream`
    (L2 flushed before each when `flush` is a buffer).  Returns the K times in
    ms and the wall-clock seconds of the timed loop."""
    import torch
    for _ in range(max(3, warmup)):
        if flush is not None:
            flush.zero_()
        fn()
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    with windows:
        t0 = time.perf_counter()
        head_start(stream)
        for a, b in ev:
            if flush is not None:
                flush.zero_()
            a.record(stream)
            fn()
            b.record(stream)
        torch.cuda.synchronize()
        wall = time.perf_counter() - t0
    return [a.elapsed_time(b) for a, b in ev], wall


def next_tree_ept(w, dev, stream, K, n_ept=4, chain=3, B=4):
    """Next-step candidate generation on trees whose every candidate carries
    n_ept ensemble chains of `chain` prompt tokens (the headline workload's
    vocabulary), with the chains' logits and then their probabilities
    averaged.  Acceptance comes from the library's argmax and acceptance
    calls.  Times each mode with CUDA events (median of K calls).  Algorithmic
    bytes: for every sequence, state k times n_ept logits rows of V fp32 (the
    rows ranked; the probability mode reads them a second time, from L2)."""
    import torch

    from paper_2405_18628_gb300 import ppd
    from paper_2405_18628_gb300 import workloads as W
    we = W.scaled(w, B=B, T=16 * (1 + n_ept * chain), n_cand=16, chains=f"ept{n_ept}x{chain}")
    s = W.make_step_inputs(we, seed=we.seed)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
    logits = torch.from_numpy(s.logits).to(dev)
    parent, cand, prefix = i32(s.parent), i32(s.cand_tokens), i32(s.prefix_len)
    o = {k: torch.empty(shape, dtype=torch.int32, device=dev) for k, shape in
         (("argmax", (we.B, we.T)), ("accept_len", (we.B,)), ("path", (we.B, we.T)),
          ("next_token", (we.B,)), ("new_prefix_len", (we.B,)), ("status", (we.B,)))}
    ws = ppd.workspace(1, we.B, 1, we.T, we.D, we.V, we.S_max, device=dev)
    ppd.ppd_node_argmax(logits, o["argmax"], workspace=ws, stream=stream)
    ppd.ppd_accept_path(o["argmax"], cand, parent, prefix, we.V, we.S_max, o["accept_len"],
                        o["path"], o["next_token"], o["new_prefix_len"], o["status"],
                        stream=stream)
    n_states, K_guess, T_next = chain + 1, 8, 64
    tp, trk = W.make_tree_templates(n_states, T_next, K_guess, np.random.default_rng(we.seed),
                                    n_ept=n_ept)
    tp_d, tr_d = i32(tp), i32(trk)
    nx = {k: torch.empty(shape, dtype=torch.int32, device=dev) for k, shape in
          (("parent", (we.B, T_next)), ("cand", (we.B, T_next)), ("state", (we.B,)),
           ("status", (we.B,)))}
    ws_nt = torch.empty(max(256, ppd.load().ppd_next_tree_workspace_bytes(we.B, n_states, K_guess)),
                        dtype=torch.uint8, device=dev)
    res = {"batch": we.B, "tree_tokens": we.T, "n_ept": n_ept, "chain_tokens": chain,
           "states": n_states, "guesses_per_depth": K_guess}
    for mode in ("logits", "probs"):
        call = lambda: ppd.ppd_next_tree(logits, parent, cand, o["path"], o["accept_len"],
                                         o["next_token"], tp_d, tr_d, K_guess, nx["parent"],
                                         nx["cand"], nx["state"], nx["status"], workspace=ws_nt,
                                         stream=stream, n_ept=n_ept, ept_mean=mode)
        for _ in range(3):
            call()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(K)]
        head_start(stream)
        for a, b in ev:
            a.record(stream)
            call()
            b.record(stream)
        torch.cuda.synchronize()
        if (o["status"].cpu().numpy() != 0).any() or (nx["status"].cpu().numpy() != 0).any():
            raise SystemExit("ensemble next-tree generation reported an error")
        us = statistics.median(a.elapsed_time(b) for a, b in ev) * 1e3
        states = nx["state"].cpu().numpy()
        nbytes = int(states.sum()) * n_ept * we.V * 4
        res[mode] = {"us": us, "state_histogram": np.bincount(states, minlength=n_states).tolist(),
                     "bytes": nbytes, "gbs": nbytes / (us * 1e-6) / 1e9}
    return res


def per_layer_attention(w, t, prefix, parent, out, dev, reps, windows):
    """Attention as a model runs it: L ppd_tree_attention calls of one layer
    each, captured in a CUDA graph and replayed `reps` times (CUDA events on the
    replay stream, median).  With a workspace the library shares each call's
    key tiles over all SMs when the layer has fewer slices than SMs; without,
    one whole slice per SM."""
    import torch

    from paper_2405_18628_gb300 import ppd

    st = torch.zeros(w.B, dtype=torch.int32, device=dev)
    ws = ppd.workspace(1, w.B, w.H, w.T, w.D, 1, w.S_max, device=dev)
    res = {}
    for mode, wsx in (("split", ws), ("unsplit", None)):
        def layers():
            for l in range(w.L):
                ppd.ppd_tree_attention(t["q"][l:l + 1], t["k_cache"][l:l + 1], t["v_cache"][l:l + 1],
                                       t["k_tree"][l:l + 1], t["v_tree"][l:l + 1], prefix, parent,
                                       out[l:l + 1], st, workspace=wsx)
        layers()
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        cap = torch.cuda.Stream()
        cap.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g, stream=cap):
                layers()
        torch.cuda.current_stream().wait_stream(cap)
        s = torch.cuda.current_stream()
        ms, _ = time_loop(g.replay, reps, 5, s, None, windows)
        if (st.cpu().numpy() != 0).any():
            raise SystemExit(f"per-layer attention reported device status {st.cpu().tolist()}")
        us = statistics.median(ms) * 1e3
        res[mode] = {"us_per_step": us, "us_per_layer": us / w.L,
                     "gbs": attention_bytes(w) / (us * 1e-6) / 1e9}
        del g
    return {"graph": True, "layers": w.L, "slices_per_layer": w.B * w.H, **res}


def copy_bandwidth(n_bytes, dev, reps=20):
    """GB/s of host-to-device and device-to-host copies of `n_bytes` between a
    pinned host buffer and device memory, each direction alone and both at
    once on two streams (median of `reps` each)."""
    import torch
    h = torch.empty(n_bytes, dtype=torch.uint8, pin_memory=True)
    d = torch.empty(n_bytes, dtype=torch.uint8, device=dev)
    h2 = torch.empty(n_bytes, dtype=torch.uint8, pin_memory=True)
    d2 = torch.empty(n_bytes, dtype=torch.uint8, device=dev)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()

    def timed(fn):
        out = []
        for _ in range(reps + 2):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            fn()
            torch.cuda.synchronize()
            out.append(time.perf_counter() - t0)
        return statistics.median(out[2:])

    def both():
        with torch.cuda.stream(s1):
            d.copy_(h, non_blocking=True)
        with torch.cuda.stream(s2):
            h2.copy_(d2, non_blocking=True)

    ss = [torch.cuda.Stream() for _ in range(4)]

    def four():
        q4 = n_bytes // 4
        for i, si in enumerate(ss):
            with torch.cuda.stream(si):
                d[i * q4:(i + 1) * q4].copy_(h[i * q4:(i + 1) * q4], non_blocking=True)

    t_in = timed(lambda: d.copy_(h, non_blocking=True))
    t_out = timed(lambda: h2.copy_(d2, non_blocking=True))
    t_both = timed(both)
    t_four = timed(four)
    return {"bytes": n_bytes, "h2d_gbs": n_bytes / t_in / 1e9, "d2h_gbs": n_bytes / t_out / 1e9,
            "both_directions_gbs": 2 * n_bytes / t_both / 1e9,
            "h2d_four_streams_gbs": (n_bytes // 4 * 4) / t_four / 1e9}


def e2e_groups(L):
    """Layer groups of the pipelined end-to-end step, in the proportions
    3 : 4 : 4 : 3 : 2 (6, 8, 8, 6, 4 of 32 layers): the first group's copy in
    overlaps no compute and the last group's compute and copy back overlap no
    copy in, so both are smaller; a group of a few layers is latency-bound
    (one call streams few tiles per SM), so neither is tiny.  Measured at
    Vicuna-7B shapes (device span of one graph replay): 424 us against 434
    for 8 / 8 / 8 / 8 and 443 for 14 / 10 / 6 / 2."""
    if L < 8:
        return [L]
    parts = [3, 4, 4, 3, 2]
    sizes = [max(1, (p * L) // 16) for p in parts]
    sizes[1] += L - sum(sizes)
    return [n for n in sizes if n > 0]


def e2e_pipelined(w, t, st, K, groups, dev, check_against=None, n_cmp=2):
    """The step end to end from pinned host buffers through the public C ABI,
    with the copies overlapping the compute.  The layers go in `groups` groups.
    Each group's Q, tree K and tree V sit together in one pinned host buffer
    and one device buffer (the tree's index arrays -- parents, candidate
    tokens, prefix lengths -- ride in front of the first group's), so a group
    is one copy in.  A group's attention (ppd_tree_attention) starts as soon
    as its copy has landed, on one of `n_cmp` compute streams in turn (so one
    group's last, partial round of slices overlaps the next group's first),
    while the next group's copy runs; its output is copied back on another
    stream as soon as it is done.  The logits come in last: node argmax
    (ppd_node_argmax) and acceptance (ppd_accept_path) need no attention
    output, so they run on a stream of their own once the logits have landed,
    then the compaction of each group's accepted rows (ppd_kv_compact; it
    writes cache rows at and past each prefix length, which no attention call
    of the step reads), and the index outputs go back after the last group's
    output.  A step ends with every
    result in host memory (stream synchronised).  Returns the timing, the
    copied bytes and, with `check_against` (the device step's outputs), the
    largest difference found."""
    import torch

    from paper_2405_18628_gb300 import ppd
    L = w.L
    if isinstance(groups, int):
        bounds = [(g * L) // groups for g in range(groups + 1)]
    else:                                   # explicit group sizes, in order
        bounds = [0]
        for n in groups:
            bounds.append(bounds[-1] + n)
        assert bounds[-1] == L
        groups = len(groups)
    tree_specs = {"parent": ((w.B, w.T), torch.int32), "cand": ((w.B, w.T), torch.int32),
                  "prefix": ((w.B,), torch.int32)}
    h_in, d_in, dv = [], [], []             # per group: host buffer, device buffer, views
    for g in range(groups):
        a, b = bounds[g], bounds[g + 1]
        specs = dict(tree_specs) if g == 0 else {}
        specs.update({k: ((b - a,) + tuple(t[k].shape[1:]), t[k].dtype)
                      for k in ("q", "k_tree", "v_tree")})
        hb, hvw = packed(specs, "cpu")
        db, dvw = packed(specs, dev)
        for k in ("q", "k_tree", "v_tree"):
            hvw[k].copy_(t[k][a:b])
        if g == 0:
            tree_h, tree_d = hvw, dvw
        h_in.append(hb)
        d_in.append(db)
        dv.append(dvw)
    tree_h["parent"].copy_(st.parent.cpu())
    tree_h["cand"].copy_(st.cand.cpu())
    tree_h["prefix"].copy_(st.prefix.cpu())
    h_logits = st.logits.cpu().pin_memory()
    d_logits = torch.empty_like(h_logits, device=dev)
    out = torch.empty(L, w.B, w.H, w.T, w.D, dtype=torch.float32, device=dev)
    h_out = torch.empty(out.shape, dtype=torch.float32, pin_memory=True)
    names = ["argmax", "accept_len", "path", "next_token", "new_prefix_len", "dev_status"]
    shapes = {"argmax": (w.B, w.T), "accept_len": (w.B,), "path": (w.B, w.T),
              "next_token": (w.B,), "new_prefix_len": (w.B,), "dev_status": (w.B,)}
    d_idx, di = packed({k: (shapes[k], torch.int32) for k in names}, dev)
    h_idx, hi = packed({k: (shapes[k], torch.int32) for k in names}, "cpu")
    st_grp = torch.zeros(groups, w.B, dtype=torch.int32, device=dev)
    # one workspace per compute stream (a call's work split keeps its partial
    # states there until its merge grid has run), one for the argmax
    ws = [st.bufs.workspace] + [torch.zeros_like(st.bufs.workspace) for _ in range(n_cmp)]
    s_in = torch.cuda.Stream()
    s_cmp = [torch.cuda.Stream() for _ in range(n_cmp)]
    s_out = torch.cuda.Stream()
    s_idx = torch.cuda.Stream()
    kc, vc = t["k_cache"], t["v_cache"]

    def one_step():
        ev_in = [torch.cuda.Event() for _ in range(groups)]
        ev_logits = torch.cuda.Event()
        ev_done = [torch.cuda.Event() for _ in range(groups)]
        ev_idx = torch.cuda.Event()
        with torch.cuda.stream(s_in):
            for g in range(groups):
                d_in[g].copy_(h_in[g], non_blocking=True)
                ev_in[g].record(s_in)
            d_logits.copy_(h_logits, non_blocking=True)
            ev_logits.record(s_in)

        # argmax and acceptance once the logits are in, then the compaction
        with torch.cuda.stream(s_idx):
            s_idx.wait_event(ev_logits)
            ppd.ppd_node_argmax(d_logits, di["argmax"], workspace=ws[n_cmp], stream=s_idx)
            ppd.ppd_accept_path(di["argmax"], tree_d["cand"], tree_d["parent"], tree_d["prefix"],
                                w.V, w.S_max, di["accept_len"], di["path"], di["next_token"],
                                di["new_prefix_len"], di["dev_status"], stream=s_idx)
            ev_idx.record(s_idx)
            for g in range(groups):
                a, b = bounds[g], bounds[g + 1]
                ppd.ppd_kv_compact(kc[a:b], vc[a:b], dv[g]["k_tree"], dv[g]["v_tree"], di["path"],
                                   di["accept_len"], tree_d["prefix"], stream=s_idx)
        for g in range(groups):
            a, b = bounds[g], bounds[g + 1]
            sc = s_cmp[g % n_cmp]
            sc.wait_event(ev_in[g])
            ppd.ppd_tree_attention(dv[g]["q"], kc[a:b], vc[a:b], dv[g]["k_tree"], dv[g]["v_tree"],
                                   tree_d["prefix"], tree_d["parent"], out[a:b], st_grp[g],
                                   workspace=ws[g % n_cmp], stream=sc)
            ev_done[g].record(sc)
            s_out.wait_event(ev_done[g])
            with torch.cuda.stream(s_out):
                h_out[a:b].copy_(out[a:b], non_blocking=True)
        s_out.wait_event(ev_idx)
        with torch.cuda.stream(s_out):
            h_idx.copy_(d_idx, non_blocking=True)

    # the copies and calls of a step captured once in a CUDA graph (the host
    # enqueues one replay per step); the side streams fork from and join the
    # capturing stream
    for _ in range(2):
        one_step()
        torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    cap = torch.cuda.Stream()
    cap.wait_stream(torch.cuda.current_stream())
    with torch.cuda.graph(graph, stream=cap):
        for x in (s_in, *s_cmp, s_out, s_idx):
            x.wait_stream(cap)
        one_step()
        for x in (s_in, *s_cmp, s_out, s_idx):
            cap.wait_stream(x)
    torch.cuda.synchronize()
    for _ in range(3):
        graph.replay()
        torch.cuda.synchronize()
    ms = []
    for _ in range(K):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        graph.replay()                            # on the current stream
        torch.cuda.current_stream().synchronize()
        ms.append((time.perf_counter() - t0) * 1e3)
    res = {"ms": ms, "h2d_bytes": int(sum(x.numel() for x in h_in) + h_logits.numel() * 4),
           "d2h_bytes": int(h_out.numel() * 4 + h_idx.numel()), "groups": groups}
    if check_against is not None:
        ref_out, ref_idx = check_against
        res["max_abs_diff_out"] = float((h_out - ref_out).abs().max())
        res["index_outputs_equal"] = all(torch.equal(hi[k], ref_idx[k]) for k in names)
        res["group_status_ok"] = bool((st_grp == 0).all().item())
    return res


def summarize(w, ms, n_acc, peak, launches):
    q10, q50, q90 = np.percentile(ms, [10, 50, 90])
    mean = float(np.mean(ms))
    sb = step_bytes(w, n_acc)
    return {"ms_per_step": mean, "ms_per_step_p10_p50_p90": [float(q10), float(q50), float(q90)],
            "steps_per_s": 1e3 / mean, "step_bytes": sb, "step_gbs": sb / (mean * 1e-3) / 1e9,
            "frac": sb / (mean * 1e-3) / 1e9 / peak,
            "frac_of_8000": sb / (mean * 1e-3) / 1e9 / NOMINAL_HBM_GBS, "launches": launches}


def rotating_inputs(w, st, K, warmup, dev, stream, accept, windows):
    """The same step timed the other way the timing rules allow for inputs
    below L2: no flush, and the step cycles over enough identical copies of its
    inputs (equal seeds, separate buffers) that each copy is read again only
    after more than 4x L2 of other copies.  The zero-fill flush leaves up to
    the whole L2 (129 MB) of dirty lines, whose write-back to HBM lands inside
    the next step; here no other write is pending when a step starts."""
    import torch
    n = int(np.ceil(4 * L2_BYTES / max(1, step_bytes(w, 0)))) + 1
    copies = [st] + [Step(w, dev, w.seed, accept) for _ in range(n - 1)]
    for c in copies[1:]:
        c(stream)
    torch.cuda.synchronize()
    for c in copies[1:]:
        c.check()
    k = [0]

    def rot():
        copies[k[0] % n](stream)
        k[0] += 1

    ms, _ = time_loop(rot, K, warmup, stream, None, windows)
    q10, q50, q90 = np.percentile(ms, [10, 50, 90])
    del copies[1:]
    torch.cuda.empty_cache()
    return {"ms_per_step": float(np.mean(ms)),
            "ms_per_step_p10_p50_p90": [float(q10), float(q50), float(q90)],
            "copies": n, "copy_bytes": int(step_bytes(w, 0)),
            "l2": f"not flushed: {n} copies of the inputs in turn "
                  f"({n * step_bytes(w, 0) / 1e6:.0f} MB, over 4x L2)"}


def bench_extra_workload(name, K, warmup, dev, stream, peak, windows, accept, with_per_layer):
    """One of the other workloads: its own inputs, K timed steps (L2 flushed
    before each when the inputs are below 4x L2), freed afterwards."""
    import torch

    from paper_2405_18628_gb300 import ppd
    from paper_2405_18628_gb300 import workloads as W
    w = W.WORKLOADS[name]
    need = 2 * w.L * w.B * w.H * (w.S_max + 2 * w.T) * w.D * 2
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    if need * 1.3 > free:
        return {"skipped": f"needs {need / 2**30:.0f} GiB of device memory"}
    st = Step(w, dev, w.seed, accept)
    flush = (torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
             if flushes_l2(w, "auto") else None)
    st(stream)
    torch.cuda.synchronize()
    n_acc = st.check()
    ms, _ = time_loop(lambda: st(stream), K, warmup, stream, flush, windows)
    n_launch = ppd.ppd_verify_step_launches(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max,
                                            typical=accept == "typical")
    res = summarize(w, ms, n_acc, peak, n_launch)
    res["l2"] = "flushed before every step" if flush is not None else "not flushed"
    if flush is not None:
        res["rotating_inputs"] = rotating_inputs(w, st, K, warmup, dev, stream, accept, windows)
    res["shape"] = {"layers": w.L, "batch": w.B, "heads": w.H, "head_dim": w.D,
                    "prefix": w.P, "tree_tokens": w.T, "vocab": w.V}
    if with_per_layer:
        res["per_layer_attention"] = per_layer_attention(w, st.t, st.prefix, st.parent,
                                                         st.bufs.out, dev, min(K, 100), windows)
    del st, flush
    torch.cuda.empty_cache()
    return res


def main(argv=None):
    args = parse(argv)
    world, rank, local = dist_setup()
    w = resolve_workload(args)
    if args.impl == "reference":
        run_reference(args, w, world, rank)
        return

    import torch
    from paper_2405_18628_gb300 import ppd

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist
    ppd.load()
    if args.form is not None:
        ppd.ppd_set_verify_step_form(args.form)
    extras = world == 1 and not args.no_extras and not args.layers
    clocks = ClockSampler(local).start()
    windows = Windows()
    peak, peak_kind = measured_peak_gbs()

    # ---------------------------------------------------------------- inputs (resident in HBM)
    seed = w.seed + 1000 * rank
    st = Step(w, dev, seed, args.accept)
    t, s, bufs, logits = st.t, st.s, st.bufs, st.logits
    parent, cand, prefix = st.parent, st.cand, st.prefix
    stream = torch.cuda.current_stream()
    do_flush = flushes_l2(w, args.l2)
    flush = torch.empty(L2_FLUSH_BYTES if do_flush else 0, dtype=torch.uint8, device=dev)

    def maybe_flush():
        if do_flush:
            flush.zero_()

    for _ in range(max(3, args.warmup)):
        maybe_flush()
        st(stream)
    torch.cuda.synchronize()
    n_acc = st.check()

    # ---------------------------------------------------------------- timed region
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    with windows:
        wall0 = time.perf_counter()
        head_start(stream)
        for k in range(K):
            maybe_flush()
            ev[k][0].record(stream)
            st(stream)
            ev[k][1].record(stream)
        torch.cuda.synchronize()
        if pg:
            pg.barrier()
        wall = time.perf_counter() - wall0
    step_ms = [a.elapsed_time(b) for a, b in ev]
    q10, q50, q90 = np.percentile(step_ms, [10, 50, 90])
    total_ms = max_over_ranks(sum(step_ms), pg, dev)
    ms_per_step = total_ms / K
    value = aggregate_rate(K, world, total_ms)

    # ---------------------------------------------------------------- dominant kernel alone
    st_att = torch.empty(w.B, dtype=torch.int32, device=dev)
    att, _ = time_loop(lambda: ppd.ppd_tree_attention(t["q"], t["k_cache"], t["v_cache"],
                                                      t["k_tree"], t["v_tree"], prefix, parent,
                                                      bufs.out, st_att, stream=stream),
                       min(K, 300), 3, stream, flush if do_flush else None, windows)
    att_ms = statistics.mean(att)
    att_bytes = attention_bytes(w)
    achieved = att_bytes / (att_ms * 1e-3) / 1e9
    tr = None if args.layers else MEASURED_TRAFFIC.get(w.name)
    traffic = tr["bytes_per_launch"] if tr and tr.get("src") == attention_source_hash() else None

    # ---------------------------------------------------------------- end to end, host buffers
    e2e = None
    if not args.no_e2e:
        K3 = min(K, 200)
        # every per-step input in one pinned host buffer and every output in one
        # device buffer, so a step is one copy in, the call, one copy out
        src_in = {"q": t["q"], "k_tree": t["k_tree"], "v_tree": t["v_tree"], "logits": logits,
                  "parent": parent, "cand": cand, "prefix": prefix}
        in_specs = {k: (v.shape, v.dtype) for k, v in src_in.items()}
        h_buf, h_in = packed(in_specs, "cpu")
        d_buf, d_in = packed(in_specs, dev)
        for k, v in src_in.items():
            h_in[k].copy_(v)
        outs = ["out", "argmax", "accept_len", "path", "next_token", "new_prefix_len", "dev_status"]
        out_specs = {k: (getattr(bufs, k).shape, getattr(bufs, k).dtype) for k in outs}
        do_buf, d_out = packed(out_specs, dev)
        ho_buf, _ = packed(out_specs, "cpu")
        h2d = h_buf.numel()
        d2h = ho_buf.numel()

        def e2e_step():
            d_buf.copy_(h_buf, non_blocking=True)
            common = (d_in["q"], t["k_cache"], t["v_cache"], d_in["k_tree"], d_in["v_tree"],
                      d_in["prefix"], d_in["parent"], d_in["cand"], d_in["logits"])
            outs_ = tuple(d_out[k] for k in outs) + (bufs.workspace,)
            if args.accept == "typical":
                ppd.ppd_verify_step_typical(*common, *TYPICAL, *outs_, stream=stream)
            else:
                ppd.ppd_verify_step(*common, *outs_, stream=stream)
            ho_buf.copy_(do_buf, non_blocking=True)
            stream.synchronize()

        for _ in range(3):
            maybe_flush()
            e2e_step()
        e_ms = []
        for _ in range(K3):
            maybe_flush()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            e2e_step()
            e_ms.append((time.perf_counter() - t0) * 1e3)
        e_total = max_over_ranks(sum(e_ms), pg, dev)
        serial = {"value": aggregate_rate(K3, world, e_total), "unit": "steps/s",
                  "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
                  "ms_per_step": e_total / K3,
                  "note": "KV cache resident on the device; per-step tree tensors, logits and "
                          "index arrays copied in from one pinned host buffer, every output "
                          "copied back into one (256-byte aligned members, one copy each way), "
                          "copies and the step one after another"}
        e2e = dict(serial)
        bw = copy_bandwidth(int(h2d), dev)
        if args.accept == "exact" and w.L >= 4:
            # the same step with the copies overlapping the compute, by layer groups;
            # checked against the device step's outputs on the same inputs
            ref = (bufs.out.cpu(), {k: getattr(bufs, k).cpu() for k in
                                    ("argmax", "accept_len", "path", "next_token", "new_prefix_len",
                                     "dev_status")})
            pip = e2e_pipelined(w, t, st, K3, e2e_groups(w.L), dev, check_against=ref)
            ok = (pip["index_outputs_equal"] and pip["group_status_ok"]
                  and pip["max_abs_diff_out"] <= 5e-3)
            p_total = max_over_ranks(sum(pip["ms"]), pg, dev)
            pipelined = {"value": aggregate_rate(K3, world, p_total), "unit": "steps/s",
                         "h2d_bytes_per_step": pip["h2d_bytes"], "d2h_bytes_per_step": pip["d2h_bytes"],
                         "ms_per_step": p_total / K3, "layer_groups": pip["groups"],
                         "matches_device_step": ok, "max_abs_diff_out": pip["max_abs_diff_out"],
                         "note": "KV cache resident on the device; the layers in groups of "
                                 + "/".join(str(n) for n in e2e_groups(w.L)) + ", each "
                                 "group's Q and tree K/V in one pinned buffer (the tree's index "
                                 "arrays in front of the first), copied in as one copy on one "
                                 "stream, its attention (ppd_tree_attention) run as soon as it "
                                 "has landed, on two compute streams in turn, its output copied "
                                 "back on a third as soon as it is done; the logits copied in "
                                 "last, then ppd_node_argmax, ppd_accept_path and ppd_kv_compact "
                                 "on a fourth stream and the index outputs copied back; the "
                                 "copies and calls of a step captured once in a CUDA graph and "
                                 "replayed once per step"}
            if ok:
                e2e = dict(pipelined)
                e2e["serial"] = serial
            else:
                e2e["pipelined_rejected"] = pipelined
        e2e["copy_gbs"] = bw

    # ---------------------------------------------------------------- next-step candidates
    next_tree = None
    if args.next_tree or extras:
        from paper_2405_18628_gb300 import workloads as W
        i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
        n_states, K_guess = 5, 8
        tp, trk = W.make_tree_templates(n_states, w.T, K_guess, np.random.default_rng(w.seed))
        tp_d, tr_d = i32(tp), i32(trk)
        nxt = {k: torch.empty(shape, dtype=torch.int32, device=dev) for k, shape in
               (("parent", (w.B, w.T)), ("cand", (w.B, w.T)), ("state", (w.B,)), ("status", (w.B,)))}
        ws_nt = torch.empty(max(256, ppd.load().ppd_next_tree_workspace_bytes(w.B, n_states, K_guess)),
                            dtype=torch.uint8, device=dev)

        def next_step():
            ppd.ppd_next_tree(logits, parent, cand, bufs.path, bufs.accept_len, bufs.next_token,
                              tp_d, tr_d, K_guess, nxt["parent"], nxt["cand"], nxt["state"],
                              nxt["status"], workspace=ws_nt, stream=stream)

        K4 = min(K, 200)
        ev4 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(K4)]
        for k in range(K4 + 3):
            st(stream)
            if k >= 3:
                ev4[k - 3][0].record(stream)
            next_step()
            if k >= 3:
                ev4[k - 3][1].record(stream)
        torch.cuda.synchronize()
        if (nxt["status"].cpu().numpy() != 0).any():
            raise SystemExit("next-step candidate generation reported an error")
        nt_ms = statistics.median(a.elapsed_time(b) for a, b in ev4)
        nt_states = nxt["state"].cpu().numpy()
        nt_bytes = int(nt_states.sum()) * w.V * 4
        next_tree = {"us": nt_ms * 1e3, "states": n_states, "guesses_per_depth": K_guess,
                     "state_histogram": np.bincount(nt_states, minlength=n_states).tolist(),
                     "bytes": nt_bytes, "gbs": nt_bytes / (nt_ms * 1e-3) / 1e9}
        if nt_bytes == 0:
            next_tree["note"] = ("state 0 for every sequence: the accepted end node of this "
                                 "workload's tree carries no prompt chain, so no guesses are "
                                 "ranked (see \"ensemble\" for a case that ranks them)")
        if extras:
            next_tree["ensemble"] = next_tree_ept(w, dev, stream, K4)

    # ---------------------------------------------------------------- typical acceptance
    typical = None
    if extras and args.accept == "exact":
        st_t = Step(w, dev, w.seed, "typical")
        ms_t, _ = time_loop(lambda: st_t(stream), min(K, 300), args.warmup, stream,
                            flush if do_flush else None, windows)
        n_acc_t = st_t.check()
        typical = summarize(w, ms_t, n_acc_t, peak,
                            ppd.ppd_verify_step_launches(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max,
                                                         typical=True))
        typical["temperature_epsilon_delta"] = list(TYPICAL)
        typical["accepted_tokens"] = n_acc_t
        del st_t
        torch.cuda.empty_cache()

    # ---------------------------------------------------------------- per-layer attention
    per_layer = None
    if extras or args.per_layer:
        per_layer = per_layer_attention(w, t, prefix, parent, bufs.out, dev, min(K, 100), windows)

    # ---------------------------------------------------------------- CPU baseline (oracle)
    cpu = None
    if world == 1 and rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, t, s, args.cpu_budget)

    sb = step_bytes(w, n_acc)
    n_launch = ppd.ppd_verify_step_launches(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max,
                                            typical=args.accept == "typical")
    del st, t, bufs, logits, flush
    torch.cuda.empty_cache()

    # ---------------------------------------------------------------- the other workloads
    others = None
    if extras:
        others = {}
        for name in EXTRA_WORKLOADS:
            others[name] = bench_extra_workload(name, K, args.warmup, dev, stream, peak, windows,
                                                args.accept, name in ("mobilellama", "vicuna13b"))

    # ---------------------------------------------------------------- tree-size profile
    profile = None
    sizes_arg = args.tree_sizes if args.tree_sizes is not None else (
        ",".join(str(n) for n in PROFILE_SIZES) if extras else "")
    if sizes_arg:
        from paper_2405_18628_gb300 import tree_profile
        sizes = [int(x) for x in sizes_arg.split(",") if x.strip()]
        lat = tree_profile.latency_profile(w, sizes, steps=max(K, 20), warmup=3, device=dev,
                                           flush_bytes=L2_FLUSH_BYTES if do_flush else 0,
                                           timed=windows)
        profile = {"base": w.name, "steps_each": max(K, 20),
                   "latency": [{"T": n, "ms_per_step": ms} for n, ms in lat]}
        if args.tau:
            from paper_2405_18628_gb300 import tree_profile as tp_
            with open(args.tau) as f:
                tau = {int(k): float(v) for k, v in json.load(f).items()}
            rows, best = tp_.speedup_table(tau, lat)
            profile["speedup"] = rows
            profile["best_tree_size"] = best

    clocks.stop()
    clk = clocks.summary(windows.spans)

    kernel = "tree_attention_kernel" if w.T <= 64 else "tree_attention_rows_kernel"
    alone = {"kernel": kernel, "launch_us": att_ms * 1e3, "bytes_per_launch": att_bytes,
             "achieved": achieved, "frac": achieved / peak}
    if n_launch == 1:
        # the whole step is one launch of the attention kernel (node argmax,
        # acceptance and compaction in its side warps): its duration is the
        # timed step, its algorithmic bytes the step's
        roof = {"bound": "hbm", "achieved": sb / (ms_per_step * 1e-3) / 1e9, "peak": peak,
                "unit": "GB/s", "traffic": traffic, "kernel": kernel + " (whole fused step)",
                "launch_us": ms_per_step * 1e3, "bytes_per_launch": sb}
    else:
        roof = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                "traffic": traffic, "kernel": kernel + " (attention alone)",
                "launch_us": att_ms * 1e3, "bytes_per_launch": att_bytes}
    roof["frac"] = roof["achieved"] / peak
    roof["peak_kind"] = peak_kind
    roof["frac_of_8000"] = roof["achieved"] / NOMINAL_HBM_GBS
    if traffic is not None:
        roof["traffic_note"] = ("ncu dram__bytes_read.sum + dram__bytes_write.sum of a 19-layer "
                                "capture scaled to all layers; output writes still in L2 at "
                                "kernel end are not counted")
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": config_of(w, args, world),
            "ms_per_step_p10_p50_p90": [float(q10), float(q50), float(q90)],
            "step_gbs": sb / (ms_per_step * 1e-3) / 1e9,
            "step_frac_of_8tbs": sb / (ms_per_step * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
            "step_bytes": sb,
            "roofline": roof,
            "attention_alone": alone,
            "e2e": e2e,
            "gpu_launches": n_launch * K,
            "form": ppd.ppd_verify_step_form(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max),
            "clocks": clk,
            "cpu_baseline": cpu,
            "wall_s_timed": wall,
        }
        if others is not None:
            line["workloads"] = others
        if per_layer is not None:
            line["per_layer_attention"] = per_layer
        if profile is not None:
            line["tree_size_profile"] = profile
        if next_tree is not None:
            line["next_tree"] = next_tree
        if typical is not None:
            line["typical_step"] = typical
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
