"""Python binding of libppd (include/ppd.h): argument marshalling only.

Each function has the name of the C entry point it calls, takes torch CUDA
tensors, derives the sizes from their shapes, and passes raw device pointers
and the current CUDA stream.  Every step of the verification path runs in the
library's kernels; there is no fallback.  A missing or unloadable library
raises immediately.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libppd.so")

PPD_OK, PPD_ERR_INVALID_ARG, PPD_ERR_UNSUPPORTED, PPD_ERR_TREE, PPD_ERR_CAPACITY, \
    PPD_ERR_CUDA, PPD_ERR_TIMEOUT = range(7)
PPD_BF16, PPD_F32 = 0, 1

_lib = None


class PPDError(RuntimeError):
    def __init__(self, status: int, where: str):
        msg = f"{where}: {status_string(status)} (status {status})"
        if status == PPD_ERR_CUDA and _lib is not None:
            msg += f", {_lib.ppd_last_cuda_error().decode()}"
        super().__init__(msg)
        self.status = status


def load() -> ctypes.CDLL:
    """Load libppd.so (built by ``paper_2405_18628_gb300.build``)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: run paper_2405_18628_gb300.build.build() "
                               "(or __graft_entry__.build()) first")
        lib = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, f32, sz = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_float,
                                 ctypes.c_size_t)
        sig = {
            "ppd_workspace_bytes": ([i32] * 7 + [i32], sz),
            "ppd_verify_step_launches": ([i32] * 7 + [i32, i32], i32),
            "ppd_verify_step_form": ([i32] * 7 + [i32], i32),
            "ppd_set_verify_step_form": ([i32], i32),
            "ppd_debug_grid_wait": ([ctypes.c_ulonglong, i32], i32),
            "ppd_status_string": ([i32], ctypes.c_char_p),
            "ppd_last_cuda_error": ([], ctypes.c_char_p),
            "ppd_last_cuda_error": ([], ctypes.c_char_p),
            "ppd_tree_attention": ([vp] * 7 + [i32] * 7 + [f32, vp, vp, vp, vp, sz, vp], i32),
            "ppd_node_argmax": ([vp, i32, i32, i32, vp, vp, sz, vp], i32),
            "ppd_accept_path": ([vp] * 4 + [i32] * 4 + [vp] * 5 + [vp], i32),
            "ppd_kv_compact": ([vp] * 7 + [i32] * 7 + [vp], i32),
            "ppd_verify_step": ([vp] * 9 + [i32] * 8 + [f32] + [vp] * 8 + [vp, sz, vp], i32),
            "ppd_selftest_umma": ([vp, vp, vp, i32, i32, vp], i32),
            "ppd_node_argmax_noalloc": ([vp, i32, i32, i32, vp, vp], i32),
            "ppd_node_stats": ([vp, i32, i32, i32, f32, vp, vp, vp, vp, sz, vp], i32),
            "ppd_typical_accept": ([vp] * 7 + [i32] * 4 + [f32] * 3 + [vp] * 5 + [vp], i32),
            "ppd_next_tree_workspace_bytes": ([i32, i32, i32], sz),
            "ppd_next_tree_ept": ([vp] * 6 + [i32] * 5 + [vp, vp, i32, i32, i32] + [vp] * 4 +
                                  [vp, sz, vp], i32),
            "ppd_next_tree": ([vp] * 6 + [i32] * 5 + [vp, vp, i32, i32] + [vp] * 4 + [vp, sz, vp],
                              i32),
            "ppd_verify_step_typical": ([vp] * 9 + [i32] * 8 + [f32] * 4 + [vp] * 8 +
                                        [vp, sz, vp], i32),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
    return _lib


def status_string(status: int) -> str:
    return load().ppd_status_string(int(status)).decode()


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libppd takes CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("libppd takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return PPD_BF16
    if t.dtype == torch.float32:
        return PPD_F32
    raise TypeError(f"q/k/v must be bfloat16 or float32, got {t.dtype}")


def _check(status: int, where: str):
    if status != PPD_OK:
        raise PPDError(status, where)


def ppd_workspace_bytes(L, B, H, T, D, V, S_max, dtype=PPD_BF16) -> int:
    return int(load().ppd_workspace_bytes(L, B, H, T, D, V, S_max, dtype))


def ppd_verify_step_launches(L, B, H, T, D, V, S_max, dtype=PPD_BF16, typical=False) -> int:
    """Kernels one ppd_verify_step (or ppd_verify_step_typical) call enqueues."""
    return int(load().ppd_verify_step_launches(L, B, H, T, D, V, S_max, dtype, int(typical)))


def ppd_verify_step_form(L, B, H, T, D, V, S_max, dtype=PPD_BF16) -> int:
    """Form of the fused step for these sizes: 0 separate grids, 1 argmax grid
    then attention grid, 2 one grid with the argmax in the side warps, 3 one
    grid with the argmax in the CTAs of the last, partial round."""
    return int(load().ppd_verify_step_form(L, B, H, T, D, V, S_max, dtype))


def ppd_set_verify_step_form(form: int) -> int:
    """Force the fused step's form (1, 2 or 3; -1 = automatic); returns the
    previous setting."""
    return int(load().ppd_set_verify_step_form(int(form)))


def ppd_debug_grid_wait(limit_ns: int, withhold_cta: int = -1) -> None:
    """Tests of the timeout path: the one-grid step's grid-wide wait gives up
    after limit_ns (0: the default 4 s) and CTA withhold_cta never publishes
    its flag (-1: none)."""
    _check(load().ppd_debug_grid_wait(int(limit_ns), int(withhold_cta)), "ppd_debug_grid_wait")


def workspace(L, B, H, T, D, V, S_max, dtype=PPD_BF16, device="cuda") -> torch.Tensor:
    """A scratch buffer of ppd_workspace_bytes(...) bytes (allocated by torch)."""
    n = ppd_workspace_bytes(L, B, H, T, D, V, S_max, dtype)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device)


def ppd_tree_attention(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, out,
                       dev_status, lse=None, scale: float = 0.0, workspace=None, stream=None):
    """q/k_tree/v_tree [L,B,H,T,D], caches [L,B,H,S_max,D], out fp32 [L,B,H,T,D]."""
    L, B, H, T, D = q.shape
    S_max = k_cache.shape[3]
    ws_n = workspace.numel() if workspace is not None else 0
    st = load().ppd_tree_attention(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(k_tree), _ptr(v_tree), _ptr(prefix_len),
        _ptr(parent), L, B, H, T, D, S_max, _dtype(q), float(scale), _ptr(out), _ptr(lse),
        _ptr(dev_status), _ptr(workspace), ws_n, _stream(stream))
    _check(st, "ppd_tree_attention")


def ppd_node_argmax(logits, argmax_out, workspace=None, stream=None):
    """logits fp32 [B,T,V] -> argmax_out int32 [B,T]."""
    B, T, V = logits.shape
    ws_n = workspace.numel() if workspace is not None else 0
    st = load().ppd_node_argmax(_ptr(logits), B, T, V, _ptr(argmax_out), _ptr(workspace), ws_n,
                                _stream(stream))
    _check(st, "ppd_node_argmax")


def ppd_node_argmax_noalloc(logits, argmax_out, stream=None):
    """Node argmax without a workspace: logits fp32 [B,T,V] -> argmax_out int32
    [B,T], partial maxima kept in the library's fixed device array."""
    B, T, V = logits.shape
    st = load().ppd_node_argmax_noalloc(_ptr(logits), B, T, V, _ptr(argmax_out), _stream(stream))
    _check(st, "ppd_node_argmax_noalloc")


def ppd_accept_path(argmax, cand_tokens, parent, prefix_len, V, S_max, accept_len, path,
                    next_token, new_prefix_len, dev_status, stream=None):
    B, T = parent.shape
    st = load().ppd_accept_path(_ptr(argmax), _ptr(cand_tokens), _ptr(parent), _ptr(prefix_len),
                                B, T, int(V), int(S_max), _ptr(accept_len), _ptr(path),
                                _ptr(next_token), _ptr(new_prefix_len), _ptr(dev_status),
                                _stream(stream))
    _check(st, "ppd_accept_path")


def ppd_kv_compact(k_cache, v_cache, k_tree, v_tree, path, accept_len, prefix_len, stream=None):
    L, B, H, S_max, D = k_cache.shape
    T = k_tree.shape[3]
    st = load().ppd_kv_compact(_ptr(k_cache), _ptr(v_cache), _ptr(k_tree), _ptr(v_tree),
                               _ptr(path), _ptr(accept_len), _ptr(prefix_len), L, B, H, T, D,
                               S_max, _dtype(k_cache), _stream(stream))
    _check(st, "ppd_kv_compact")


def ppd_verify_step(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                    logits, out, argmax_out, accept_len, path, next_token, new_prefix_len,
                    dev_status, workspace, lse=None, scale: float = 0.0, stream=None):
    L, B, H, T, D = q.shape
    S_max = k_cache.shape[3]
    V = logits.shape[2]
    st = load().ppd_verify_step(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(k_tree), _ptr(v_tree), _ptr(prefix_len),
        _ptr(parent), _ptr(cand_tokens), _ptr(logits), L, B, H, T, D, V, S_max, _dtype(q),
        float(scale), _ptr(out), _ptr(lse), _ptr(argmax_out), _ptr(accept_len), _ptr(path),
        _ptr(next_token), _ptr(new_prefix_len), _ptr(dev_status), _ptr(workspace),
        workspace.numel(), _stream(stream))
    _check(st, "ppd_verify_step")


def ppd_node_stats(logits, temperature: float, argmax_out, lse_out, entropy_out, workspace,
                   stream=None):
    """logits fp32 [B,T,V] -> argmax int32 [B,T], log-sum-exp and entropy fp32
    [B,T] of softmax(logits / temperature)."""
    B, T, V = logits.shape
    st = load().ppd_node_stats(_ptr(logits), B, T, V, float(temperature), _ptr(argmax_out),
                               _ptr(lse_out), _ptr(entropy_out), _ptr(workspace),
                               workspace.numel(), _stream(stream))
    _check(st, "ppd_node_stats")


def ppd_typical_accept(logits, lse, entropy, argmax, cand_tokens, parent, prefix_len, S_max,
                       temperature: float, epsilon: float, delta: float, accept_len, path,
                       next_token, new_prefix_len, dev_status, stream=None):
    B, T, V = logits.shape
    st = load().ppd_typical_accept(
        _ptr(logits), _ptr(lse), _ptr(entropy), _ptr(argmax), _ptr(cand_tokens), _ptr(parent),
        _ptr(prefix_len), B, T, V, int(S_max), float(temperature), float(epsilon), float(delta),
        _ptr(accept_len), _ptr(path), _ptr(next_token), _ptr(new_prefix_len), _ptr(dev_status),
        _stream(stream))
    _check(st, "ppd_typical_accept")


def ppd_verify_step_typical(q, k_cache, v_cache, k_tree, v_tree, prefix_len, parent, cand_tokens,
                            logits, temperature: float, epsilon: float, delta: float, out,
                            argmax_out, accept_len, path, next_token, new_prefix_len, dev_status,
                            workspace, lse=None, scale: float = 0.0, stream=None):
    L, B, H, T, D = q.shape
    S_max = k_cache.shape[3]
    V = logits.shape[2]
    st = load().ppd_verify_step_typical(
        _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(k_tree), _ptr(v_tree), _ptr(prefix_len),
        _ptr(parent), _ptr(cand_tokens), _ptr(logits), L, B, H, T, D, V, S_max, _dtype(q),
        float(scale), float(temperature), float(epsilon), float(delta), _ptr(out), _ptr(lse),
        _ptr(argmax_out), _ptr(accept_len), _ptr(path), _ptr(next_token), _ptr(new_prefix_len),
        _ptr(dev_status), _ptr(workspace), workspace.numel(), _stream(stream))
    _check(st, "ppd_verify_step_typical")


def ppd_next_tree(logits, parent, cand_tokens, path, accept_len, next_token, tmpl_parent,
                  tmpl_rank, K: int, next_parent, next_cand, next_state, dev_status,
                  workspace=None, stream=None, n_ept: int = 1, ept_mean: str = "logits"):
    """Next-step candidate tree.  logits [B,T,V]; parent, cand_tokens, path
    [B,T]; accept_len, next_token [B]; tmpl_parent, tmpl_rank [n_states,
    T_next] (device int32); n_ept ensemble prompt tokens per prompt position,
    whose logits (ept_mean="logits") or probabilities ("probs") are averaged;
    outputs next_parent, next_cand [B,T_next], next_state, dev_status [B].  A
    workspace is allocated if none is given."""
    if ept_mean not in ("logits", "probs"):
        raise ValueError(f"ept_mean must be 'logits' or 'probs', not {ept_mean!r}")
    B, T, V = logits.shape
    n_states, T_next = tmpl_parent.shape
    need = int(load().ppd_next_tree_workspace_bytes(B, n_states, int(K)))
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=logits.device)
    st = load().ppd_next_tree_ept(_ptr(logits), _ptr(parent), _ptr(cand_tokens), _ptr(path),
                                  _ptr(accept_len), _ptr(next_token), B, T, V, n_states, T_next,
                                  _ptr(tmpl_parent), _ptr(tmpl_rank), int(K), int(n_ept),
                                  int(ept_mean == "probs"), _ptr(next_parent), _ptr(next_cand),
                                  _ptr(next_state), _ptr(dev_status), _ptr(workspace),
                                  workspace.numel(), _stream(stream))
    _check(st, "ppd_next_tree")


def ppd_selftest_umma(a, b, d, mode: int, N: int, stream=None):
    st = load().ppd_selftest_umma(_ptr(a), _ptr(b), _ptr(d), int(mode), int(N), _stream(stream))
    _check(st, "ppd_selftest_umma")


class StepBuffers:
    """Device outputs and workspace of one verification step for given sizes."""

    def __init__(self, L, B, H, T, D, V, S_max, dtype=PPD_BF16, device="cuda", with_lse=False):
        i32 = dict(dtype=torch.int32, device=device)
        self.out = torch.empty((L, B, H, T, D), dtype=torch.float32, device=device)
        self.lse = torch.empty((L, B, H, T), dtype=torch.float32, device=device) if with_lse else None
        self.argmax = torch.empty((B, T), **i32)
        self.accept_len = torch.empty(B, **i32)
        self.path = torch.empty((B, T), **i32)
        self.next_token = torch.empty(B, **i32)
        self.new_prefix_len = torch.empty(B, **i32)
        self.dev_status = torch.empty(B, **i32)
        self.workspace = workspace(L, B, H, T, D, V, S_max, dtype, device)
