#!/usr/bin/env python3
"""Benchmark of the PPD verification step (tree attention over every layer,
node argmax, acceptance, KV compaction) through libppd's C ABI.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl reference]

Prints one JSON line.  The default workload is the Vicuna-7B-shaped cache
(32 layers, 32 heads x 128, bf16 K/V, batch 1, prefix 2048, 64-token tree,
vocab 32000).  Inputs are seeded synthetic tensors resident in HBM.  When a
step's inputs are at least four times the 129 MB L2 (every Vicuna-shaped
workload: 1.17 GB per step at Vicuna-7B), steps run back to back and no step
can find the previous one's data in L2; smaller workloads flush L2 (a 256 MiB
write) before every timed step, outside the step's events.

Under torchrun (N > 1) each rank runs an independent replica of the workload
on its own GPU (weak scaling: the sequences of different ranks are
independent, no data-path collective); the step time is the maximum over
ranks.  `--impl reference` times the fp64 CPU oracle on the host cores
instead (rank 0 only), on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
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

# DRAM traffic of one launch of the roofline kernel (dram__bytes_read.sum +
# dram__bytes_write.sum), keyed by workload, with the hash of the attention
# sources it was taken on: a stale entry reports null.  The captures ran the
# same shapes with 19 layers (608 / 760 units: whole rounds of 152 CTAs) and
# are scaled to the full layer count, since traffic grows with the units
# (the logits, read once per step, are not scaled).
MEASURED_TRAFFIC = {
    # whole fused step: 685,382,912 B at 19 layers; slices x 32/19, logits once
    "vicuna7b": {"bytes_per_launch": 1_148_724_062, "src": "34ce1a8dc4edf4e2"},
    # whole fused step: 1,672,942,592 B at 19 layers; slices x 40/19, logits once
    "vicuna13b": {"bytes_per_launch": 3_508_402_931, "src": "34ce1a8dc4edf4e2"},
}


def attention_source_hash() -> str:
    h = hashlib.sha256()
    for f in ("ppd_attention.cu", "ppd_attention_rows.cu", "ppd_attention_common.cuh",
              "ppd_device.cuh", "ppd_accept.cuh", "ppd_kernels.h", "ppd_api.cu"):
        with open(os.path.join(ROOT, "paper_2405_18628_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def per_layer_attention(w, t, prefix, parent, out, dev, reps):
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
        for _ in range(5):
            g.replay()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for a, b in ev:
            a.record(s)
            g.replay()
            b.record(s)
        torch.cuda.synchronize()
        if (st.cpu().numpy() != 0).any():
            raise SystemExit(f"per-layer attention reported device status {st.cpu().tolist()}")
        us = statistics.median(a.elapsed_time(b) for a, b in ev) * 1e3
        res[mode] = {"us_per_step": us, "us_per_layer": us / w.L,
                     "gbs": attention_bytes(w) / (us * 1e-6) / 1e9}
        del g
    return {"graph": True, "layers": w.L, "slices_per_layer": w.B * w.H, **res}


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
    the compacted K/V rows (read from the tree, written to the cache) and the
    small integer arrays."""
    ints = 4 * w.B * w.T * 4 + 4 * w.B * 6
    return (attention_bytes(w) + 4 * w.B * w.T * w.V +
            2 * 4 * w.L * w.H * w.D * n_acc_total + ints)


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) >= 9 and parts[1].replace(".", "").isdigit():
                        rows.append(parts)
        except Exception:
            pass
        finally:
            if self.path and os.path.exists(self.path):
                os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[k] for r in rows for k in range(4) if r[5 + k].lower() == "active"})
        return {"sm_mhz": statistics.median(float(r[1]) for r in rows),
                "sm_max_mhz": max(float(r[2]) for r in rows),
                "power_w_max": max(float(r[3]) for r in rows if r[3].replace(".", "").isdigit())
                if any(r[3].replace(".", "").isdigit() for r in rows) else None,
                "reasons": reasons, "samples": len(rows)}


# ----------------------------------------------------------------------------- CPU oracle

def oracle_step_seconds(w, host, s, units, n_threads: int) -> float:
    """One fp64 oracle verification step on a sample of the workload, scaled to
    the whole step.  `host` holds the first few layers of Q/K/V on the host;
    attention runs on `units` of them (None: all), compaction on all of them,
    argmax and acceptance once, as in a full step.  Attention and compaction
    times are scaled by the fraction of the workload the sample covers."""
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


def cpu_baseline(w, t_dev, s, budget_s: float):
    """Oracle on the first `nl` layers, `nl` chosen from a one-layer calibration
    so the sample takes about `budget_s` seconds of host time."""
    import oracle
    n_threads = os.cpu_count() or 1
    one = {k: v[:1].cpu() for k, v in t_dev.items()}
    t0 = time.perf_counter()
    oracle_step_seconds(w, one, s, None, n_threads)
    t1 = time.perf_counter() - t0
    nl = max(1, min(w.L, int(budget_s / max(t1, 1e-6))))
    host = one if nl == 1 else {k: v[:nl].cpu() for k, v in t_dev.items()}
    sec = oracle_step_seconds(w, host, s, None, n_threads)
    return {"value": 1.0 / sec, "unit": "steps/s", "cores": n_threads, "kind": "oracle",
            "sample": f"fp64 oracle verification step on the first {nl} of {w.L} layers "
                      f"(all heads; attention and compaction time scaled by {w.L}/{nl}; "
                      f"full argmax and acceptance)"}


# ----------------------------------------------------------------------------- main

def parse():
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
    ap.add_argument("--accept", default="exact", choices=["exact", "typical"],
                    help="verification rule: exact matching, or typical acceptance at "
                         "temperature 0.7, epsilon 0.09, delta 0.3")
    ap.add_argument("--tree-sizes", default="",
                    help="comma-separated tree sizes: also report the step latency of each "
                         "(the hardware half of the paper's hardware-aware tree size)")
    ap.add_argument("--tau", default="",
                    help="JSON file {tree size: acceptance length}: with --tree-sizes, also "
                         "report Speedup(n) = tau(n) / latency(n) and the best size")
    ap.add_argument("--next-tree", action="store_true",
                    help="also time next-step candidate generation (ppd_next_tree, 5 tree "
                         "states, 8 guesses per depth) after each step")
    ap.add_argument("--per-layer", action="store_true",
                    help="also time the attention as it runs inside a model: one "
                         "ppd_tree_attention call per layer, the L calls captured in a CUDA graph")
    ap.add_argument("--layers", type=int, default=0,
                    help="run the workload with this many layers (profiling captures)")
    ap.add_argument("--l2", default="auto", choices=["auto", "flush", "none"],
                    help="auto: flush L2 before each step unless the step's inputs exceed 4x L2")
    return ap.parse_args()


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


def run_reference(args, w, world, rank):
    """The CPU oracle as the reference arm.  Each step is a bounded sample: a
    few attention slices of layer 0 (scaled to all slices), the full argmax and
    acceptance, and layer 0's compaction (scaled to all layers)."""
    if rank != 0:
        return
    from paper_2405_18628_gb300 import workloads as W

    s = W.make_step_inputs(w)
    n_threads = os.cpu_count() or 1
    host = W.make_tensors(W.scaled(w, L=1), device="cpu")
    n_all = w.B * w.H
    cal = list(range(min(n_threads, n_all)))
    t0 = time.perf_counter()
    oracle_step_seconds(w, host, s, cal, n_threads)
    t_cal = time.perf_counter() - t0
    per_step_budget = max(0.01, 150.0 / max(1, args.steps + args.warmup))
    n_units = int(max(1, min(n_all, len(cal) * per_step_budget / max(t_cal, 1e-9))))
    units = list(range(n_units))
    for _ in range(args.warmup):
        oracle_step_seconds(w, host, s, units, n_threads)
    secs = [oracle_step_seconds(w, host, s, units, n_threads) for _ in range(args.steps)]
    sec_per_step = statistics.mean(secs)
    value = 1.0 / sec_per_step
    sample = (f"{n_units} of {w.L * w.B * w.H} attention slices (layer 0) per step, scaled to all "
              f"slices; full argmax and acceptance; layer-0 compaction scaled to {w.L} layers")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": "steps/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": sec_per_step * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name},
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": n_threads, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }), flush=True)


def main():
    args = parse()
    world, rank, local = dist_setup()
    from paper_2405_18628_gb300 import workloads as W
    w = W.WORKLOADS[args.config]
    if args.layers:
        # fewer layers of the same shapes: small cases for profiler captures
        w = W.scaled(w, L=args.layers)
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

    # ---------------------------------------------------------------- inputs (resident in HBM)
    s = W.make_step_inputs(w, seed=w.seed + 1000 * rank)
    t = W.make_tensors(w, device=dev, seed=w.seed + 1000 * rank)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
    parent, cand, prefix = i32(s.parent), i32(s.cand_tokens), i32(s.prefix_len)
    logits = torch.from_numpy(s.logits).to(dev)
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
    stream = torch.cuda.current_stream()
    footprint = step_bytes(w, 0)
    do_flush = args.l2 == "flush" or (args.l2 == "auto" and footprint < 4 * L2_BYTES)
    flush = torch.empty(L2_FLUSH_BYTES if do_flush else 0, dtype=torch.uint8, device=dev)

    def maybe_flush():
        if do_flush:
            flush.zero_()

    def step():
        if args.accept == "typical":
            ppd.ppd_verify_step_typical(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                        prefix, parent, cand, logits, *TYPICAL, bufs.out,
                                        bufs.argmax, bufs.accept_len, bufs.path, bufs.next_token,
                                        bufs.new_prefix_len, bufs.dev_status, bufs.workspace,
                                        stream=stream)
        else:
            ppd.ppd_verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"], prefix,
                                parent, cand, logits, bufs.out, bufs.argmax, bufs.accept_len,
                                bufs.path, bufs.next_token, bufs.new_prefix_len, bufs.dev_status,
                                bufs.workspace, stream=stream)

    for _ in range(max(3, args.warmup)):
        maybe_flush()
        step()
    torch.cuda.synchronize()
    status = bufs.dev_status.cpu().numpy()
    n_acc = int(bufs.accept_len.sum().item())
    if (status != 0).any() or n_acc < w.B:
        raise SystemExit(f"verification step reported device status {status.tolist()}")

    # ---------------------------------------------------------------- timed region
    K = args.steps
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(K)]
    with ClockSampler(local) as clocks:
        if pg:
            pg.barrier()
        torch.cuda.synchronize()
        wall0 = time.perf_counter()
        for k in range(K):
            maybe_flush()
            ev[k][0].record(stream)
            step()
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
    clk = clocks.summary()

    # ---------------------------------------------------------------- dominant kernel alone
    K2 = min(K, 300)
    ev2 = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(K2)]
    st_att = torch.empty(w.B, dtype=torch.int32, device=dev)
    for k in range(K2 + 3):
        maybe_flush()
        if k >= 3:
            ev2[k - 3][0].record(stream)
        ppd.ppd_tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"], prefix,
                               parent, bufs.out, st_att, stream=stream)
        if k >= 3:
            ev2[k - 3][1].record(stream)
    torch.cuda.synchronize()
    att_ms = statistics.mean(a.elapsed_time(b) for a, b in ev2)
    att_bytes = attention_bytes(w)
    peak, peak_kind = measured_peak_gbs()
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
        e2e = {"value": aggregate_rate(K3, world, e_total), "unit": "steps/s",
               "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
               "ms_per_step": e_total / K3,
               "note": "KV cache resident on the device; per-step tree tensors, logits and "
                       "index arrays copied in from one pinned host buffer, every output "
                       "copied back into one (256-byte aligned members, one copy each way)"}

    # ---------------------------------------------------------------- CPU baseline (oracle)
    cpu = None
    if world == 1 and rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, t, s, args.cpu_budget)

    # ---------------------------------------------------------------- next-step candidates
    next_tree = None
    if args.next_tree:
        n_states, K_guess = 5, 8
        tp, tr = W.make_tree_templates(n_states, w.T, K_guess, np.random.default_rng(w.seed))
        tp_d, tr_d = i32(tp), i32(tr)
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
            step()
            if k >= 3:
                ev4[k - 3][0].record(stream)
            next_step()
            if k >= 3:
                ev4[k - 3][1].record(stream)
        torch.cuda.synchronize()
        if (nxt["status"].cpu().numpy() != 0).any():
            raise SystemExit("next-step candidate generation reported an error")
        nt_ms = statistics.median(a.elapsed_time(b) for a, b in ev4)
        next_tree = {"us": nt_ms * 1e3, "states": n_states, "guesses_per_depth": K_guess,
                     "state_histogram": np.bincount(nxt["state"].cpu().numpy(),
                                                    minlength=n_states).tolist()}

    # ---------------------------------------------------------------- per-layer attention
    per_layer = None
    if args.per_layer:
        per_layer = per_layer_attention(w, t, prefix, parent, bufs.out, dev, min(K, 100))

    # ---------------------------------------------------------------- tree-size profile
    profile = None
    if args.tree_sizes:
        from paper_2405_18628_gb300 import tree_profile
        del t, bufs, logits
        torch.cuda.empty_cache()
        sizes = [int(x) for x in args.tree_sizes.split(",") if x.strip()]
        lat = tree_profile.latency_profile(w, sizes, steps=min(K, 50), warmup=3, device=dev,
                                           flush_bytes=L2_FLUSH_BYTES if do_flush else 0)
        profile = {"latency": [{"T": n, "ms_per_step": ms} for n, ms in lat]}
        if args.tau:
            with open(args.tau) as f:
                tau = {int(k): float(v) for k, v in json.load(f).items()}
            rows, best = tree_profile.speedup_table(tau, lat)
            profile["speedup"] = rows
            profile["best_tree_size"] = best

    sb = step_bytes(w, n_acc)
    n_launch = ppd.ppd_verify_step_launches(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max,
                                            typical=args.accept == "typical")
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
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "steps/s", "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name + (f" ({w.L} layers)" if args.layers else ""),
                       "layers": w.L, "batch": w.B, "heads": w.H,
                       "head_dim": w.D, "prefix": w.P, "tree_tokens": w.T, "vocab": w.V,
                       "S_max": w.S_max,
                       "l2": ("flushed before every step (256 MiB write, outside the step events)"
                              if do_flush else
                              f"not flushed: inputs larger than L2 ({footprint / 1e6:.0f} MB "
                              f"streamed per step, L2 {L2_BYTES / 1e6:.0f} MB)"),
                       "parallelism": f"replicas x{world}",
                       "accept": ("exact matching" if args.accept == "exact" else
                                  "typical acceptance (temperature %g, epsilon %g, delta %g)"
                                  % TYPICAL)},
            "ms_per_step_p10_p50_p90": [float(q10), float(q50), float(q90)],
            "step_gbs": sb / (ms_per_step * 1e-3) / 1e9,
            "step_frac_of_8tbs": sb / (ms_per_step * 1e-3) / 1e9 / NOMINAL_HBM_GBS,
            "step_bytes": sb,
            "roofline": roof,
            "attention_alone": alone,
            "e2e": e2e,
            "gpu_launches": n_launch * K,
            "clocks": clk,
            "cpu_baseline": cpu,
            "wall_s_timed": wall,
        }
        if profile is not None:
            line["tree_size_profile"] = profile
        if next_tree is not None:
            line["next_tree"] = next_tree
        if per_layer is not None:
            line["per_layer_attention"] = per_layer
        print(json.dumps(line), flush=True)
    if pg:
        pg.barrier()
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
