"""The attention work split against the oracle.  Launches with fewer slices
than SMs share all key tiles out over every SM, and the slices cut between
SMs are merged by a second grid.

Cases: calls with few slices and long prefixes (many parts per slice);
prefixes far shorter than the cache (fewer tiles than SMs, so some SMs get
none); both kernels, including trees over 128 tokens; launches with more
slices than SMs (whole slices, with a workspace).  Also: the unsplit path (no
workspace), repeated calls on one workspace, and a workspace full of junk
(any contents must do)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

from test_gpu_parity import assert_attn_close, i32, tensors

pytestmark = pytest.mark.gpu

def _case(L, B, H, T, D, prefix, S_max, seed):
    rng = np.random.default_rng(seed)
    parent = np.full((B, T), -1, np.int32)
    for b in range(B):
        for i in range(1, T):
            parent[b, i] = rng.integers(0, i)
    w = W.Workload("split", L=L, B=B, H=H, D=D, P=S_max, T=T, V=16, n_cand=T, max_depth=T,
                   chains="every0", match_rate=0.5, seed=seed)
    pl = np.asarray(prefix, np.int32)
    t = tensors(w, prefix_len=pl)
    return t, pl, parent


def _attend(t_dev, pl, parent, dev, ws):
    L, B, H, T, D = t_dev["q"].shape
    out = torch.full((L, B, H, T, D), float("nan"), device=dev)
    lse = torch.full((L, B, H, T), float("nan"), device=dev)
    st = torch.full((B,), -7, dtype=torch.int32, device=dev)
    ppd.ppd_tree_attention(t_dev["q"], t_dev["k_cache"], t_dev["v_cache"], t_dev["k_tree"],
                           t_dev["v_tree"], i32(pl, dev), i32(parent, dev), out, st, lse=lse,
                           workspace=ws)
    torch.cuda.synchronize()
    return out.cpu().numpy(), lse.cpu().numpy(), st.cpu().numpy()


CASES = [
    # L, B, H, T, D, prefix, S_max: what it exercises (all split but the last two)
    (1, 1, 2, 64, 128, [3000], 3072),          # 2 slices x 25 tiles over 50 SMs: 25 parts each
    (2, 3, 5, 48, 64, [0, 129, 2000], 2048),   # mixed prefixes, empty prefix, D = 64
    (1, 2, 3, 40, 128, [100, 5], 4096),        # 12 tiles for 152 SMs: empty ranges
    (1, 1, 2, 96, 128, [2500], 2560),          # query-row kernel, slices cut many times
    (1, 2, 1, 200, 128, [900, 33], 1024),      # two query blocks and two tree tiles per slice
    (1, 1, 1, 512, 64, [300], 1024),           # four query blocks, tree tiles alone in a part
    (2, 1, 32, 64, 128, [2048], 2112),         # Vicuna-7B shapes, two layers
    (2, 1, 100, 64, 128, [700], 768),          # 200 slices: whole slices round-robin
    (1, 2, 80, 96, 128, [300, 1000], 1024),    # query-row kernel, 160 slices: round-robin
]


@pytest.mark.parametrize("L,B,H,T,D,prefix,S_max", CASES)
def test_split_matches_oracle(cuda_device, L, B, H, T, D, prefix, S_max):
    t, pl, parent = _case(L, B, H, T, D, prefix, S_max, seed=L * 100 + T + D)
    t_dev = {k: v.to(cuda_device) for k, v in t.items()}
    ref, ref_lse, _, ref_st = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                                    t["v_tree"], pl, parent)
    assert (ref_st == 0).all()
    ws = ppd.workspace(L, B, H, T, D, 1, S_max, device=cuda_device)
    for rep in range(2):                       # the workspace is reusable
        out, lse, st = _attend(t_dev, pl, parent, cuda_device, ws)
        assert (st == 0).all(), st
        assert_attn_close(out.reshape(ref.shape), ref, f"split, call {rep}")
        np.testing.assert_allclose(lse.reshape(ref_lse.shape), ref_lse, rtol=0, atol=1e-3)
    # the unsplit path: one whole slice per SM at a time
    out, lse, st = _attend(t_dev, pl, parent, cuda_device, None)
    assert (st == 0).all()
    assert_attn_close(out.reshape(ref.shape), ref, "unsplit")


def test_split_in_fused_step(cuda_device):
    """The fused verification step with slices cut between SMs: attention
    within tolerance, indices and compacted KV bit for bit."""
    w = W.scaled(W.WORKLOADS["mobilellama"], L=2, H=3)
    s = W.make_step_inputs(w)
    t = tensors(w, prefix_len=s.prefix_len)
    dev = cuda_device
    td = {k: v.to(dev) for k, v in t.items()}
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
    ppd.ppd_verify_step(td["q"], td["k_cache"], td["v_cache"], td["k_tree"], td["v_tree"],
                        i32(s.prefix_len, dev), i32(s.parent, dev), i32(s.cand_tokens, dev),
                        torch.from_numpy(s.logits).to(dev), bufs.out, bufs.argmax,
                        bufs.accept_len, bufs.path, bufs.next_token, bufs.new_prefix_len,
                        bufs.dev_status, bufs.workspace)
    torch.cuda.synchronize()
    ref = oracle.verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                             s.prefix_len, s.parent, s.cand_tokens, s.logits)
    assert (bufs.dev_status.cpu().numpy() == 0).all()
    assert_attn_close(bufs.out.cpu().numpy().reshape(ref["out"].shape), ref["out"], "fused")
    for k in ("argmax", "accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    for k in ("k_cache", "v_cache"):
        np.testing.assert_array_equal(td[k].cpu().view(torch.int16).numpy().view(np.uint16), ref[k],
                                      err_msg=k)


def test_workspace_contents_do_not_matter(cuda_device):
    """A workspace full of junk (NaN bit patterns, stale records) gives the
    same results: every call writes what it later reads."""
    L, B, H, T, D, prefix, S_max = CASES[0]
    t, pl, parent = _case(L, B, H, T, D, prefix, S_max, seed=5)
    t_dev = {k: v.to(cuda_device) for k, v in t.items()}
    ws = ppd.workspace(L, B, H, T, D, 1, S_max, device=cuda_device)
    ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                         t["v_tree"], pl, parent)
    for fill in (0xFF, 0x7F, 0x00):
        ws.fill_(fill)
        out, _, st = _attend(t_dev, pl, parent, cuda_device, ws)
        assert (st == 0).all()
        assert_attn_close(out.reshape(ref.shape), ref, f"workspace filled with {fill:#x}")


def test_split_status_per_call(cuda_device):
    """Per-sequence status on the split path: a malformed tree and a prefix
    beyond the cache are reported over a status array holding junk, and the
    next call on the same workspace, with clean inputs, reports neither and
    matches the oracle."""
    L, B, H, T, D, S_max = 1, 3, 2, 48, 64, 2048
    t, pl, parent = _case(L, B, H, T, D, [2000, 1500, 2000], S_max, seed=11)
    t_dev = {k: v.to(cuda_device) for k, v in t.items()}
    ws = ppd.workspace(L, B, H, T, D, 1, S_max, device=cuda_device)
    bad_parent = parent.copy()
    bad_parent[1, 5] = 7            # not before its child
    bad_pl = pl.copy()
    bad_pl[2] = t["k_cache"].shape[3] + 1   # beyond the cache
    _, _, st = _attend(t_dev, bad_pl, bad_parent, cuda_device, ws)
    assert st.tolist() == [0, ppd.PPD_ERR_TREE, ppd.PPD_ERR_CAPACITY]
    ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                         t["v_tree"], pl, parent)
    out, _, st = _attend(t_dev, pl, parent, cuda_device, ws)
    assert (st == 0).all(), st
    assert_attn_close(out.reshape(ref.shape), ref, "clean call after a failed one")
