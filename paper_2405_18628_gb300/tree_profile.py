"""Hardware-aware tree size (paper Section 4.2): the speedup of a tree budget n
is Speedup(n) = tau(n) / L_fp(n), the acceptance length over the forward-pass
latency, and the budget to use is the n that maximises it.  tau(n) depends on
the model and data only and is measured once elsewhere; L_fp(n) depends on the
hardware.  This module measures the hardware part on this GPU -- the latency of
the verification step (tree attention over every layer, node argmax,
acceptance, compaction) for each tree size -- and combines it with a
caller-supplied tau table.

The latency is that of this library's step alone, not of a whole model
forward pass; a caller who adds the rest of the forward pass passes its
latency per tree size as `extra_ms`.
"""
from __future__ import annotations

import dataclasses
import statistics
from typing import Dict, Iterable, List, Optional, Tuple

import numpy as np

from . import workloads as W


def tree_size_workload(base: W.Workload, n: int) -> W.Workload:
    """`base` with an n-token tree: ceil(n / 4) candidate nodes (the root
    included, depth capped as in `base`) and prompt-token chains of up to three
    tokens filling the rest, the shape of the paper's sparse trees."""
    if n < 1:
        raise ValueError("tree size must be positive")
    n_cand = max(1, (n + 3) // 4)
    return dataclasses.replace(base, name=f"{base.name}_n{n}", T=n, n_cand=n_cand, chains="fill3")


def measure_step_latency(w: W.Workload, steps: int = 30, warmup: int = 5, device="cuda",
                         flush_bytes: int = 0, timed=None) -> float:
    """Median device time (ms) of ppd_verify_step on workload `w`, CUDA events
    on the current stream, `warmup` untimed steps first.  With flush_bytes > 0
    a buffer of that size is written before every step (outside the events).
    `timed`, when given, is a context manager entered around the timed loop."""
    import contextlib

    import torch

    from . import ppd

    dev = torch.device(device)
    s = W.make_step_inputs(w)
    t = W.make_tensors(w, device=dev)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)
    parent, cand, prefix = i32(s.parent), i32(s.cand_tokens), i32(s.prefix_len)
    logits = torch.from_numpy(s.logits).to(dev)
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
    flush = torch.empty(flush_bytes, dtype=torch.uint8, device=dev) if flush_bytes else None
    stream = torch.cuda.current_stream()

    def step():
        ppd.ppd_verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"], prefix,
                            parent, cand, logits, bufs.out, bufs.argmax, bufs.accept_len,
                            bufs.path, bufs.next_token, bufs.new_prefix_len, bufs.dev_status,
                            bufs.workspace, stream=stream)

    for _ in range(warmup):
        if flush is not None:
            flush.zero_()
        step()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(steps)]
    torch.cuda.synchronize()
    with (timed if timed is not None else contextlib.nullcontext()):
        # a ~1 ms spin first, outside the events, so that the host has queued the
        # first steps before the GPU reaches them
        torch.cuda._sleep(2_000_000)
        for a, b in ev:
            if flush is not None:
                flush.zero_()
            a.record(stream)
            step()
            b.record(stream)
        torch.cuda.synchronize()
    status = bufs.dev_status.cpu().numpy()
    if (status != 0).any():
        raise RuntimeError(f"verification step reported device status {status.tolist()}")
    ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    del t, bufs, logits, flush
    torch.cuda.empty_cache()
    return ms


def latency_profile(base: W.Workload, sizes: Iterable[int], steps: int = 30, warmup: int = 5,
                    device="cuda", flush_bytes: int = 0, timed=None) -> List[Tuple[int, float]]:
    """L_fp(n) of the verification step on this GPU for each tree size n, as
    (n, median ms per step) pairs in the order given."""
    return [(int(n), measure_step_latency(tree_size_workload(base, int(n)), steps, warmup,
                                          device, flush_bytes, timed))
            for n in sizes]


def speedup_table(tau: Dict[int, float], latency: Iterable[Tuple[int, float]],
                  extra_ms: Optional[Dict[int, float]] = None):
    """Speedup(n) = tau(n) / L_fp(n) for every n present in both, with L_fp(n)
    the measured step latency plus extra_ms[n] (the rest of the forward pass,
    when the caller has it).  Returns (rows, best_n): rows are dicts with n,
    tau, latency_ms and speedup (accepted tokens per ms), best_n the n with the
    largest speedup (the smallest such n on ties), or None if nothing matched."""
    rows = []
    for n, ms in latency:
        if n not in tau:
            continue
        lat = ms + (extra_ms or {}).get(n, 0.0)
        if not lat > 0:
            raise ValueError(f"latency for n={n} must be positive")
        rows.append({"n": n, "tau": float(tau[n]), "latency_ms": lat, "speedup": tau[n] / lat})
    best = None
    for r in rows:
        if best is None or r["speedup"] > best["speedup"] or (
                r["speedup"] == best["speedup"] and r["n"] < best["n"]):
            best = r
    return rows, (best["n"] if best else None)
