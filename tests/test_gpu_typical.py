"""Typical acceptance on the GPU (through the C ABI) against the fp64 oracle:
node softmax statistics within float tolerance, acceptance outputs bit for bit
where every candidate's test is decided by a clear margin (checked on the
oracle's values before comparing), and the whole step with typical acceptance
(single fused grid for B <= 64, separate grids above)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

from test_gpu_parity import assert_attn_close, i32, tensors

pytestmark = pytest.mark.gpu

TEMP, EPS, DELTA = 0.7, 0.09, 0.3
MARGIN = 1e-3          # relative gap p_tok vs threshold that float rounding cannot cross


def _node_stats(logits, temp, dev):
    B, T, V = logits.shape
    x = torch.from_numpy(logits).to(dev)
    am = torch.full((B, T), -1, dtype=torch.int32, device=dev)
    lse = torch.full((B, T), float("nan"), device=dev)
    ent = torch.full((B, T), float("nan"), device=dev)
    ws = ppd.workspace(1, B, 1, T, 64, V, 1, device=dev)
    ppd.ppd_node_stats(x, temp, am, lse, ent, ws)
    torch.cuda.synchronize()
    return x, am, lse, ent


@pytest.mark.parametrize("B,T,V,temp", [(1, 64, 32000, 0.7), (3, 17, 1001, 1.3), (2, 5, 4, 0.25)])
def test_node_stats_match_oracle(cuda_device, B, T, V, temp):
    rng = np.random.default_rng(V + B)
    logits = (rng.standard_normal((B, T, V)) * 1.5).astype(np.float32)
    logits[0, 0, V - 1] = -np.inf
    if T > 2:
        logits[0, 1, min(3, V - 1)] = np.nan
        logits[-1, 2, :] = 0.25                    # uniform row: H = log V
    _, am, lse, ent = _node_stats(logits, temp, cuda_device)
    ref_lse, ref_ent = oracle.node_stats(logits, temp)
    np.testing.assert_array_equal(am.cpu().numpy(), oracle.node_argmax(logits))
    got_l, got_e = lse.cpu().numpy().astype(np.float64), ent.cpu().numpy().astype(np.float64)
    nan = np.isnan(ref_lse)
    assert (np.isnan(got_l) == nan).all() and (np.isnan(got_e) == nan).all()
    np.testing.assert_allclose(got_l[~nan], ref_lse[~nan], rtol=2e-6, atol=2e-5)
    np.testing.assert_allclose(got_e[~nan], ref_ent[~nan], rtol=2e-5, atol=2e-5)


def _margins_clear(ref):
    ratio = ref["p_tok"] / ref["threshold"]
    return np.nanmin(np.abs(ratio - 1.0)) > MARGIN


@pytest.mark.parametrize("name,overrides", [("tiny", {"B": 4}), ("mobilellama", {"L": 1, "H": 1}),
                                            ("vicuna7b", {"L": 1, "H": 1, "B": 2})])
def test_typical_accept_matches_oracle(cuda_device, name, overrides):
    w = W.scaled(W.WORKLOADS[name], **overrides)
    s = W.make_step_inputs(w)
    dev = cuda_device
    x, am, lse, ent = _node_stats(s.logits, TEMP, dev)
    ref = oracle.typical_accept(s.logits, oracle.node_argmax(s.logits), s.cand_tokens, s.parent,
                                s.prefix_len, w.S_max, TEMP, EPS, DELTA)
    assert _margins_clear(ref)
    B, T = s.parent.shape
    out = {k: torch.full((B,), -9, dtype=torch.int32, device=dev)
           for k in ("accept_len", "next_token", "new_prefix_len", "status")}
    out["path"] = torch.full((B, T), -9, dtype=torch.int32, device=dev)
    ppd.ppd_typical_accept(x, lse, ent, am, i32(s.cand_tokens, dev), i32(s.parent, dev),
                           i32(s.prefix_len, dev), w.S_max, TEMP, EPS, DELTA, out["accept_len"],
                           out["path"], out["next_token"], out["new_prefix_len"], out["status"])
    torch.cuda.synchronize()
    for k in ("accept_len", "path", "next_token", "new_prefix_len", "status"):
        np.testing.assert_array_equal(out[k].cpu().numpy(), ref[k], err_msg=k)


@pytest.mark.parametrize("name,overrides", [("tiny", {}), ("tiny", {"B": 4}),
                                            ("mobilellama", {"L": 2, "H": 4}),
                                            ("vicuna13b", {"L": 1, "H": 2})])
def test_verify_step_typical_matches_oracle(cuda_device, name, overrides):
    w = W.scaled(W.WORKLOADS[name], **overrides)
    s = W.make_step_inputs(w)
    t = tensors(w, prefix_len=s.prefix_len)
    _check_step(w, s, t, cuda_device)


@pytest.mark.parametrize("B", [64, 65])
def test_verify_step_typical_batch_paths(cuda_device, B):
    """B <= 64: the fused step; larger batches: separate grids."""
    w = W.Workload("batch", L=1, B=B, H=2, D=64, P=40, T=16, V=300, n_cand=8, max_depth=3,
                   chains="every1", match_rate=0.8, seed=B + 7)
    rng = np.random.default_rng(B)
    pl = rng.integers(0, 41, size=B).astype(np.int32)
    s = W.make_step_inputs(w, prefix_len=pl)
    t = tensors(w, prefix_len=pl)
    _check_step(w, s, t, cuda_device)


def _check_step(w, s, t, dev):
    ref = oracle.verify_step_typical(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                     s.prefix_len, s.parent, s.cand_tokens, s.logits, TEMP, EPS,
                                     DELTA)
    assert _margins_clear(ref)
    g = {k: v.to(dev) for k, v in t.items()}
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
    ppd.ppd_verify_step_typical(g["q"], g["k_cache"], g["v_cache"], g["k_tree"], g["v_tree"],
                                i32(s.prefix_len, dev), i32(s.parent, dev),
                                i32(s.cand_tokens, dev), torch.from_numpy(s.logits).to(dev),
                                TEMP, EPS, DELTA, bufs.out, bufs.argmax, bufs.accept_len,
                                bufs.path, bufs.next_token, bufs.new_prefix_len, bufs.dev_status,
                                bufs.workspace)
    torch.cuda.synchronize()
    assert_attn_close(bufs.out.cpu().numpy().reshape(ref["out"].shape), ref["out"], w.name)
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), ref["argmax"])
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), ref["status"])
    np.testing.assert_array_equal(g["k_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["k_cache"])
    np.testing.assert_array_equal(g["v_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["v_cache"])
