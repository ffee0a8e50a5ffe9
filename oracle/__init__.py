"""ctypes wrapper of the fp64 CPU oracle (``ppd_oracle.c``).

TEST INFRASTRUCTURE: only the tests, the smoke check and the benchmark's
CPU-baseline / reference arm use this package.  It shares no code with the
CUDA implementation and must never be imported by the product path.

Every function takes host arrays (numpy, or CPU torch tensors) and returns
numpy arrays.  bf16 tensors are passed as their raw 16-bit patterns; fp32
tensors are rounded to bf16 inside the C code.
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess
import sys
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ppd_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile ppd_oracle.c into liboracle.so next to it (OpenMP if available)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        raise RuntimeError("no C compiler found to build the oracle")
    tmp = _LIB + f".tmp{os.getpid()}"
    base = [cc, "-O2", "-std=c11", "-shared", "-fPIC", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        i32p = ctypes.POINTER(ctypes.c_int32)
        f64p = ctypes.POINTER(ctypes.c_double)
        i64p = ctypes.POINTER(ctypes.c_int64)
        vp = ctypes.c_void_p
        c_int, c_i64 = ctypes.c_int, ctypes.c_int64
        lib.oracle_round_bf16.argtypes = [vp, vp, c_i64]
        lib.oracle_round_bf16.restype = None
        lib.oracle_tree_attention.argtypes = [vp, vp, vp, vp, vp, c_int, i32p, i32p,
                                              c_int, c_int, c_int, c_int, c_int, c_int,
                                              ctypes.c_double, i64p, c_i64, f64p, f64p, f64p,
                                              i32p, c_int]
        lib.oracle_tree_attention.restype = c_int
        lib.oracle_node_argmax.argtypes = [vp, c_i64, c_i64, i32p]
        lib.oracle_node_argmax.restype = None
        lib.oracle_accept_path.argtypes = [i32p, i32p, i32p, i32p, c_int, c_int, c_int, c_int,
                                           i32p, i32p, i32p, i32p, i32p]
        lib.oracle_accept_path.restype = c_int
        lib.oracle_kv_compact.argtypes = [vp, vp, vp, vp, i32p, i32p, i32p, c_int, c_int,
                                          c_int, c_int, c_int, c_int, c_int]
        lib.oracle_kv_compact.restype = c_int
        c_dbl = ctypes.c_double
        lib.oracle_node_stats.argtypes = [vp, c_i64, c_i64, c_dbl, f64p, f64p]
        lib.oracle_node_stats.restype = None
        lib.oracle_typical_accept.argtypes = [vp, i32p, i32p, i32p, i32p, c_int, c_int, c_int,
                                              c_int, c_dbl, c_dbl, c_dbl, i32p, i32p, i32p, i32p,
                                              i32p, f64p, f64p]
        lib.oracle_typical_accept.restype = c_int
        lib.oracle_topk.argtypes = [vp, c_i64, c_i64, c_int, i32p]
        lib.oracle_topk.restype = None
        lib.oracle_next_tree.argtypes = [vp, i32p, i32p, i32p, i32p, i32p, c_int, c_int, c_int,
                                         c_int, c_int, i32p, i32p, c_int, c_int, i32p, i32p, i32p,
                                         i32p]
        lib.oracle_next_tree.restype = c_int
        lib.oracle_next_tree_ept.argtypes = [vp, i32p, i32p, i32p, i32p, i32p, c_int, c_int, c_int,
                                             c_int, c_int, i32p, i32p, c_int, c_int, c_int, i32p,
                                             i32p, i32p, i32p]
        lib.oracle_next_tree_ept.restype = c_int
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = c_int
        _lib = lib
    return _lib


def max_threads() -> int:
    return int(_load().oracle_max_threads())


# ----------------------------------------------------------------------------- helpers

def _host(x):
    """numpy view of a host array; bf16 torch tensors become uint16 bit patterns."""
    if isinstance(x, np.ndarray):
        return np.ascontiguousarray(x), None
    import torch
    if isinstance(x, torch.Tensor):
        if x.device.type != "cpu":
            raise ValueError("oracle inputs must be host tensors")
        x = x.contiguous()
        if x.dtype == torch.bfloat16:
            return x.view(torch.int16).numpy().view(np.uint16), "bf16"
        return x.numpy(), None
    return np.ascontiguousarray(np.asarray(x)), None


def _dtype_code(arr: np.ndarray, tag) -> int:
    if tag == "bf16" or arr.dtype == np.uint16:
        return 0
    if arr.dtype == np.float32:
        return 1
    raise TypeError(f"attention inputs must be bf16 bit patterns or float32, got {arr.dtype}")


def _i32(x):
    a, _ = _host(x)
    return np.ascontiguousarray(a, dtype=np.int32)


def _ptr(a: np.ndarray, ctype=None):
    if ctype is None:
        return ctypes.c_void_p(a.ctypes.data)
    return a.ctypes.data_as(ctypes.POINTER(ctype))


# ----------------------------------------------------------------------------- API

def round_bf16(x) -> np.ndarray:
    """fp32 -> bf16 bit patterns (uint16), round to nearest even."""
    a = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    out = np.empty(a.shape, np.uint16)
    _load().oracle_round_bf16(_ptr(a), _ptr(out), a.size)
    return out


def tree_attention(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent,
                   scale: float = 0.0, units=None, n_threads: int = 0):
    """Tree-masked attention in fp64.

    q, k_tree, v_tree: [L,B,H,T,D]; k_cache, v_cache: [L,B,H,S_max,D] (bf16 or
    fp32); prefix_len int32[B]; parent int32[B,T].  `units` optionally lists
    the (l*B+b)*H+h slices to compute.  Returns (out [n,T,D], lse [n,T],
    rowsum [n,T], status [B]) with n = len(units) or L*B*H.
    """
    arrs = [_host(t) for t in (q, k_cache, v_cache, k_tree, v_tree)]
    codes = {_dtype_code(a, tag) for a, tag in arrs}
    if len(codes) != 1:
        raise TypeError("q/k/v must share one storage type")
    dtype = codes.pop()
    qa = arrs[0][0]
    L, B, H, T, D = qa.shape
    S_max = arrs[1][0].shape[3]
    pl = _i32(prefix_len)
    par = _i32(parent)
    if units is None:
        n = L * B * H
        up = None
    else:
        ua = np.ascontiguousarray(np.asarray(units, dtype=np.int64))
        n = ua.size
        up = _ptr(ua, ctypes.c_int64)
    out = np.empty((n, T, D), np.float64)
    lse = np.empty((n, T), np.float64)
    rowsum = np.empty((n, T), np.float64)
    status = np.empty(B, np.int32)
    rc = _load().oracle_tree_attention(
        *[_ptr(a) for a, _ in arrs], dtype, _ptr(pl, ctypes.c_int32), _ptr(par, ctypes.c_int32),
        L, B, H, T, D, S_max, float(scale), up, n,
        _ptr(out, ctypes.c_double), _ptr(lse, ctypes.c_double), _ptr(rowsum, ctypes.c_double),
        _ptr(status, ctypes.c_int32), int(n_threads))
    if rc != 0:
        raise ValueError(f"oracle_tree_attention rejected its arguments (code {rc})")
    return out, lse, rowsum, status


def node_argmax(logits) -> np.ndarray:
    """argmax over the last axis of fp32 logits (first max / first NaN wins)."""
    a, _ = _host(logits)
    a = np.ascontiguousarray(a, dtype=np.float32)
    V = a.shape[-1]
    rows = a.size // V if V else 0
    out = np.empty(a.shape[:-1], np.int32)
    _load().oracle_node_argmax(_ptr(a), rows, V, _ptr(out, ctypes.c_int32))
    return out


def accept_path(argmax, cand_tokens, parent, prefix_len, V: int, S_max: int):
    """Exact-matching acceptance.  Returns dict of accept_len, path, next_token,
    new_prefix_len, status (all int32 numpy arrays)."""
    am, cd, par, pl = _i32(argmax), _i32(cand_tokens), _i32(parent), _i32(prefix_len)
    B, T = par.shape
    res = {k: np.empty(B, np.int32) for k in ("accept_len", "next_token", "new_prefix_len", "status")}
    res["path"] = np.empty((B, T), np.int32)
    p = lambda a: _ptr(a, ctypes.c_int32)
    rc = _load().oracle_accept_path(p(am), p(cd), p(par), p(pl), B, T, int(V), int(S_max),
                                    p(res["accept_len"]), p(res["path"]), p(res["next_token"]),
                                    p(res["new_prefix_len"]), p(res["status"]))
    if rc != 0:
        raise ValueError(f"oracle_accept_path rejected its arguments (code {rc})")
    return res


def node_stats(logits, temperature: float):
    """lse and entropy (fp64 numpy arrays of logits.shape[:-1]) of
    softmax(logits / temperature) over the last axis."""
    a, _ = _host(logits)
    a = np.ascontiguousarray(a, dtype=np.float32)
    V = a.shape[-1]
    rows = a.size // V if V else 0
    lse = np.empty(a.shape[:-1], np.float64)
    ent = np.empty(a.shape[:-1], np.float64)
    _load().oracle_node_stats(_ptr(a), rows, V, float(temperature), _ptr(lse, ctypes.c_double),
                              _ptr(ent, ctypes.c_double))
    return lse, ent


def typical_accept(logits, argmax, cand_tokens, parent, prefix_len, S_max: int,
                   temperature: float, epsilon: float, delta: float):
    """Typical acceptance.  logits [B,T,V] fp32.  Returns dict of accept_len,
    path, next_token, new_prefix_len, status (int32) and p_tok, threshold
    ([B,T] fp64, NaN where no test applies)."""
    lg, _ = _host(logits)
    lg = np.ascontiguousarray(lg, dtype=np.float32)
    am, cd, par, pl = _i32(argmax), _i32(cand_tokens), _i32(parent), _i32(prefix_len)
    B, T = par.shape
    V = lg.shape[-1]
    res = {k: np.empty(B, np.int32) for k in ("accept_len", "next_token", "new_prefix_len", "status")}
    res["path"] = np.empty((B, T), np.int32)
    res["p_tok"] = np.empty((B, T), np.float64)
    res["threshold"] = np.empty((B, T), np.float64)
    p = lambda a: _ptr(a, ctypes.c_int32)
    d = lambda a: _ptr(a, ctypes.c_double)
    rc = _load().oracle_typical_accept(
        _ptr(lg), p(am), p(cd), p(par), p(pl), B, T, int(V), int(S_max), float(temperature),
        float(epsilon), float(delta), p(res["accept_len"]), p(res["path"]), p(res["next_token"]),
        p(res["new_prefix_len"]), p(res["status"]), d(res["p_tok"]), d(res["threshold"]))
    if rc != 0:
        raise ValueError(f"oracle_typical_accept rejected its arguments (code {rc})")
    return res


def topk(logits, K: int) -> np.ndarray:
    """The K best tokens of each row (last axis) of fp32 logits, in ranking
    order: NaN first (lower index first), then larger value, then lower index."""
    a, _ = _host(logits)
    a = np.ascontiguousarray(a, dtype=np.float32)
    V = a.shape[-1]
    rows = a.size // V if V else 0
    out = np.empty(a.shape[:-1] + (K,), np.int32)
    _load().oracle_topk(_ptr(a), rows, V, int(K), _ptr(out, ctypes.c_int32))
    return out


def next_tree(logits, parent, cand_tokens, path, accept_len, next_token, tmpl_parent, tmpl_rank,
              K: int, n_ept: int = 1, ept_mean: str = "logits"):
    """Next-step candidate tree.  logits [B,T,V]; parent, cand_tokens, path
    [B,T]; accept_len, next_token [B]; tmpl_parent, tmpl_rank [n_states,
    T_next]; n_ept ensemble prompt tokens per position, whose logits
    (ept_mean="logits") or probabilities (ept_mean="probs") are averaged.
    Returns dict of next_parent, next_cand [B,T_next], next_state, status [B]."""
    if ept_mean not in ("logits", "probs"):
        raise ValueError(f"ept_mean must be 'logits' or 'probs', not {ept_mean!r}")
    lg, _ = _host(logits)
    lg = np.ascontiguousarray(lg, dtype=np.float32)
    par, cd, pth, al, nt = (_i32(x) for x in (parent, cand_tokens, path, accept_len, next_token))
    tp, tr = _i32(tmpl_parent), _i32(tmpl_rank)
    B, T = par.shape
    V = lg.shape[-1]
    n_states, T_next = tp.shape
    res = {"next_parent": np.empty((B, T_next), np.int32), "next_cand": np.empty((B, T_next), np.int32),
           "next_state": np.empty(B, np.int32), "status": np.empty(B, np.int32)}
    p = lambda a: _ptr(a, ctypes.c_int32)
    rc = _load().oracle_next_tree_ept(_ptr(lg), p(par), p(cd), p(pth), p(al), p(nt), B, T, V,
                                      n_states, T_next, p(tp), p(tr), int(K), int(n_ept),
                                      int(ept_mean == "probs"), p(res["next_parent"]),
                                      p(res["next_cand"]), p(res["next_state"]), p(res["status"]))
    if rc != 0:
        raise ValueError(f"oracle_next_tree rejected its arguments (code {rc})")
    return res


def kv_compact(k_cache, v_cache, k_tree, v_tree, path, accept_len, prefix_len):
    """Returns new (k_cache, v_cache) numpy copies with the accepted rows written."""
    kc, tagk = _host(k_cache)
    vc, _ = _host(v_cache)
    kt, _ = _host(k_tree)
    vt, _ = _host(v_tree)
    kc = kc.copy()
    vc = vc.copy()
    L, B, H, S_max, D = kc.shape
    T = kt.shape[3]
    pth, al, pl = _i32(path), _i32(accept_len), _i32(prefix_len)
    p = lambda a: _ptr(a, ctypes.c_int32)
    rc = _load().oracle_kv_compact(_ptr(kc), _ptr(vc), _ptr(kt), _ptr(vt), p(pth), p(al), p(pl),
                                   L, B, H, T, D, S_max, kc.itemsize)
    if rc != 0:
        raise ValueError(f"oracle_kv_compact met an out-of-range row (code {rc})")
    return kc, vc


def verify_step(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                logits, scale: float = 0.0, units=None, n_threads: int = 0):
    """The whole verification step: attention, node argmax, acceptance and
    compaction, composed in that order."""
    out, lse, rowsum, att_status = tree_attention(q, k_cache, v_cache, k_tree, v_tree,
                                                  prefix_len, parent, scale, units, n_threads)
    am = node_argmax(logits)
    S_max = _host(k_cache)[0].shape[3]
    V = _host(logits)[0].shape[-1]
    acc = accept_path(am, cand_tokens, parent, prefix_len, V, S_max)
    kc, vc = kv_compact(k_cache, v_cache, k_tree, v_tree, acc["path"], acc["accept_len"],
                        prefix_len)
    return dict(out=out, lse=lse, rowsum=rowsum, argmax=am, k_cache=kc, v_cache=vc, **acc)


def verify_step_typical(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                        logits, temperature: float, epsilon: float, delta: float,
                        scale: float = 0.0, units=None, n_threads: int = 0):
    """The verification step with typical acceptance instead of exact matching:
    attention, node argmax, typical acceptance and compaction, in that order."""
    out, lse, rowsum, att_status = tree_attention(q, k_cache, v_cache, k_tree, v_tree,
                                                  prefix_len, parent, scale, units, n_threads)
    am = node_argmax(logits)
    S_max = _host(k_cache)[0].shape[3]
    acc = typical_accept(logits, am, cand_tokens, parent, prefix_len, S_max, temperature,
                         epsilon, delta)
    kc, vc = kv_compact(k_cache, v_cache, k_tree, v_tree, acc["path"], acc["accept_len"],
                        prefix_len)
    return dict(out=out, lse=lse, rowsum=rowsum, argmax=am, k_cache=kc, v_cache=vc, **acc)
