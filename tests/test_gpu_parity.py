"""GPU path (through the C ABI) against the fp64 CPU oracle on the same seeded
inputs.  Indices, paths and compacted KV are compared bit for bit; attention
outputs within max-abs 5e-3 and relative-L2 1e-3 (fp32 outputs from the same
bf16 inputs)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ATOL = 5e-3
RTOL_L2 = 1e-3


def i32(a, dev):
    return torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(dev)


def assert_attn_close(got, ref, what=""):
    got = np.asarray(got, np.float64)
    assert np.isfinite(got).all(), f"{what}: non-finite outputs"
    err = np.abs(got - ref).max()
    rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
    assert err <= ATOL and rel <= RTOL_L2, f"{what}: max-abs {err:.3e} rel-L2 {rel:.3e}"


def run_attention(t_dev, prefix_len, parent, dev, lse=True, scale=0.0, dtype=ppd.PPD_BF16):
    q = t_dev["q"]
    L, B, H, T, D = q.shape
    S = t_dev["k_cache"].shape[3]
    out = torch.full((L, B, H, T, D), float("nan"), device=dev)
    lse_t = torch.full((L, B, H, T), float("nan"), device=dev) if lse else None
    st = torch.full((B,), -7, dtype=torch.int32, device=dev)
    ws = ppd.workspace(L, B, H, T, D, 1, S, dtype, dev)
    ppd.ppd_tree_attention(q, t_dev["k_cache"], t_dev["v_cache"], t_dev["k_tree"], t_dev["v_tree"],
                           i32(prefix_len, dev), i32(parent, dev), out, st, lse=lse_t,
                           scale=scale, workspace=ws)
    torch.cuda.synchronize()
    return out, lse_t, st


def tensors(w, seed=None, prefix_len=None):
    t = W.make_tensors(w, device="cpu", seed=seed)
    if prefix_len is not None:
        W.poison_cache_tail(t["k_cache"], t["v_cache"], prefix_len)
    return t


# ----------------------------------------------------------------------------- attention

@pytest.mark.parametrize("name,overrides,prefix", [
    ("tiny", {}, None),
    ("tiny", {"B": 3, "H": 2}, [0, 37, 300]),              # empty, ragged, multi-tile prefix
    ("mobilellama", {"L": 1, "H": 4, "P": 512}, None),
    ("vicuna7b", {"L": 1, "H": 3, "B": 2}, [2048, 1999]),
    ("vicuna13b", {"L": 1, "H": 2}, [700]),                 # T = 96
    ("sweep_t16", {"L": 1, "B": 2, "H": 2, "P": 300}, [300, 1]),
    ("sweep_t128", {"L": 1, "B": 2, "H": 2, "P": 260}, [260, 129]),
])
def test_attention_matches_oracle(cuda_device, name, overrides, prefix):
    w = W.scaled(W.WORKLOADS[name], **overrides)
    pl = np.full(w.B, w.P, np.int32) if prefix is None else np.asarray(prefix, np.int32)
    w = W.scaled(w, P=int(pl.max()))
    s = W.make_step_inputs(w, prefix_len=pl)
    t = tensors(w, prefix_len=pl)
    out, lse, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, s.parent,
                                 cuda_device)
    ref, ref_lse, _, ref_st = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                                    t["v_tree"], pl, s.parent)
    assert (st.cpu().numpy() == 0).all() and (ref_st == 0).all()
    assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, name)
    np.testing.assert_allclose(lse.cpu().numpy().reshape(ref_lse.shape), ref_lse, rtol=0,
                               atol=1e-3)


def test_attention_f32_inputs(cuda_device):
    w = W.WORKLOADS["tiny_f32"]
    s = W.make_step_inputs(w)
    t = tensors(w)
    out, _, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, s.prefix_len,
                               s.parent, cuda_device, dtype=ppd.PPD_F32)
    ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                         t["v_tree"], s.prefix_len, s.parent)
    assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, "tiny_f32")


@pytest.mark.parametrize("T,P", [(1, 0), (1, 5), (128, 0), (33, 128), (64, 4096)])
def test_attention_edge_sizes(cuda_device, T, P):
    rng = np.random.default_rng(T * 1000 + P)
    B, H, D = 2, 2, 128
    parent = np.full((B, T), -1, np.int32)
    for b in range(B):
        for i in range(1, T):
            parent[b, i] = rng.integers(0, i) if b else i - 1     # random tree / chain
    w = W.Workload("edge", L=1, B=B, H=H, D=D, P=P, T=T, V=16, n_cand=T, max_depth=T,
                   chains="every0", match_rate=0.5, seed=T + P)
    pl = np.full(B, P, np.int32)
    t = tensors(w, prefix_len=pl)
    out, _, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, parent, cuda_device)
    ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                         t["v_tree"], pl, parent)
    assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, f"T={T} P={P}")


@pytest.mark.parametrize("big", [2.0e5, 50.0])
def test_attention_values_beyond_f16(cuda_device, big):
    """Large V values in the query-row kernel (trees of 65..128 tokens, P as
    bf16 hi + lo, fp32 accumulation): a prefix tile, the last (partial) prefix
    tile and the tree tile scaled up.  With values up to 2e5 (beyond the f16
    range) the bound is 5e-3 max-abs and 1e-3 rel-L2 relative to each slice's
    magnitude: fp32 rounding alone gives an output of 2e5 an error of ~0.01.
    With values up to 50 the plain 5e-3 max-abs bound applies."""
    w = W.scaled(W.WORKLOADS["vicuna13b"], L=1, H=2, P=700)
    pl = np.array([700], np.int32)
    s = W.make_step_inputs(w, prefix_len=pl)
    t = tensors(w, prefix_len=pl)
    vc = t["v_cache"].float()
    vc[0, 0, 0, 130:140] *= big                      # head 0, second prefix tile
    vc[0, 0, 1, 650, :7] = -0.35 * big               # head 1, last (partial) prefix tile
    t["v_cache"] = vc.to(torch.bfloat16)
    vt = t["v_tree"].float()
    vt[0, 0, 1, 5] *= 0.5 * big                      # head 1, tree tile
    t["v_tree"] = vt.to(torch.bfloat16)
    out, _, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, s.parent,
                               cuda_device)
    ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                         t["v_tree"], pl, s.parent)
    got = out.cpu().numpy().reshape(ref.shape).astype(np.float64)
    assert np.isfinite(got).all()
    if big <= 1e3:
        assert_attn_close(got, ref, f"values up to {big}")
        return
    for u in range(ref.shape[0]):                    # per slice, relative to its magnitude
        scale = np.abs(ref[u]).max()
        assert np.abs(got[u] - ref[u]).max() <= 5e-3 * max(scale, 1.0), u
        assert np.linalg.norm(got[u] - ref[u]) <= 1e-3 * np.linalg.norm(ref[u]), u


@pytest.mark.parametrize("T,P", [(100, 300), (65, 128)])
def test_attention_rows_head_dim_64(cuda_device, T, P):
    """The 65..128-token kernel with 64-wide heads."""
    rng = np.random.default_rng(T + P)
    B, H, D = 2, 3, 64
    parent = np.full((B, T), -1, np.int32)
    for b in range(B):
        for i in range(1, T):
            parent[b, i] = rng.integers(0, i)
    w = W.Workload("rows64", L=1, B=B, H=H, D=D, P=P, T=T, V=16, n_cand=T, max_depth=T,
                   chains="every0", match_rate=0.5, seed=T * 7 + P)
    pl = np.array([P, P // 3], np.int32)
    t = tensors(w, prefix_len=pl)
    out, lse, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, parent,
                                 cuda_device)
    ref, ref_lse, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                               t["v_tree"], pl, parent)
    assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, f"D=64 T={T}")
    np.testing.assert_allclose(lse.cpu().numpy().reshape(ref_lse.shape), ref_lse, rtol=0,
                               atol=1e-3)


@pytest.mark.parametrize("T,P,D", [(200, 700, 128), (285, 300, 128), (512, 130, 128),
                                   (129, 0, 64), (300, 256, 64)])
def test_attention_trees_over_128_tokens(cuda_device, T, P, D):
    """Trees above 128 tokens (the paper's MobileLlama trees reach 285): query
    rows in blocks of 128, tree keys in tiles of 128, masks from 512-bit
    ancestor sets."""
    rng = np.random.default_rng(T * 31 + P + D)
    B, H = 2, 2
    parent = np.full((B, T), -1, np.int32)
    for b in range(B):
        for i in range(1, T):
            # long chains mixed with branching: ancestors across every tree tile
            parent[b, i] = i - 1 if (b == 0 and i % 5) else rng.integers(max(0, i - 150), i)
    w = W.Workload("big", L=1, B=B, H=H, D=D, P=P, T=T, V=16, n_cand=T, max_depth=T,
                   chains="every0", match_rate=0.5, seed=T + P + D)
    pl = np.array([P, max(P - 77, 0)], np.int32)
    t = tensors(w, prefix_len=pl)
    out, lse, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, parent,
                                 cuda_device)
    ref, ref_lse, _, ref_st = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                                    t["v_tree"], pl, parent)
    assert (st.cpu().numpy() == 0).all() and (ref_st == 0).all()
    assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, f"T={T} P={P} D={D}")
    np.testing.assert_allclose(lse.cpu().numpy().reshape(ref_lse.shape), ref_lse, rtol=0,
                               atol=1e-3)


def test_attention_peaked_scores_and_scale(cuda_device):
    """Large scores force the running-max rescale path on later tiles."""
    w = W.scaled(W.WORKLOADS["vicuna7b"], L=1, H=2, P=1000)
    s = W.make_step_inputs(w)
    t = tensors(w, prefix_len=s.prefix_len)
    t["q"] = (t["q"].float() * 4).to(torch.bfloat16)
    ramp = torch.linspace(0.2, 3.0, w.S_max).view(1, 1, 1, -1, 1)
    t["k_cache"] = (t["k_cache"].float() * ramp).to(torch.bfloat16)   # later tiles score higher
    for scale in (0.0, 0.3):
        out, _, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, s.prefix_len,
                                   s.parent, cuda_device, scale=scale)
        ref, _, _, _ = oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                             t["v_tree"], s.prefix_len, s.parent, scale=scale)
        assert_attn_close(out.cpu().numpy().reshape(ref.shape), ref, f"peaked scale={scale}")


def test_attention_malformed_tree_status(cuda_device):
    w = W.scaled(W.WORKLOADS["tiny"], B=3)
    s = W.make_step_inputs(w)
    parent = s.parent.copy()
    parent[1, 5] = 7            # not before its child
    pl = s.prefix_len.copy()
    pl[2] = w.S_max + 1         # beyond the cache
    t = tensors(w)
    _, _, st = run_attention({k: v.to(cuda_device) for k, v in t.items()}, pl, parent, cuda_device)
    assert st.cpu().tolist() == [0, ppd.PPD_ERR_TREE, ppd.PPD_ERR_CAPACITY]


# ----------------------------------------------------------------------------- argmax

@pytest.mark.parametrize("B,T,V", [(1, 48, 1024), (1, 64, 32000), (3, 7, 1001), (2, 128, 32000),
                                   (1, 1, 1)])
def test_node_argmax_matches_oracle(cuda_device, B, T, V):
    rng = np.random.default_rng(B * T + V)
    x = rng.standard_normal((B, T, V)).astype(np.float32)
    flat = x.reshape(B * T, V)
    if V > 10:
        for r in range(0, B * T, 3):                 # planted ties, NaNs, signed zeros
            k = rng.integers(0, V, size=3)
            kind = r % 4
            if kind == 0:
                flat[r, k] = 50.0
            elif kind == 1:
                flat[r, k[1:]] = np.nan
            elif kind == 2:
                flat[r] = -1.0
                flat[r, k[0]] = -0.0
                flat[r, k[1]] = 0.0
            else:
                flat[r] = 7.0
    out = torch.empty((B, T), dtype=torch.int32, device=cuda_device)
    ws = ppd.workspace(1, B, 1, T, 64, V, 1, device=cuda_device)
    for _ in range(2):                               # counters left clean for the next call
        out.fill_(-5)
        ppd.ppd_node_argmax(torch.from_numpy(x).to(cuda_device), out, ws)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(out.cpu().numpy(), oracle.node_argmax(x))


# ----------------------------------------------------------------------------- accept

def _random_accept_case(rng, B, T, V, match=0.6):
    parent = np.zeros((B, T), np.int32)
    cand = np.zeros((B, T), np.int32)
    top = rng.integers(0, V, size=(B, T)).astype(np.int32)
    for b in range(B):
        parent[b, 0] = -1
        cand[b, 0] = rng.integers(0, V)
        for i in range(1, T):
            parent[b, i] = rng.integers(max(0, i - 6), i) if rng.random() < 0.7 else rng.integers(0, i)
            u = rng.random()
            cand[b, i] = top[b, parent[b, i]] if u < match else (-1 if u < match + 0.2 else rng.integers(0, V))
    return parent, cand, top


@pytest.mark.parametrize("T", [1, 2, 7, 48, 64, 96, 128])
def test_accept_path_matches_oracle(cuda_device, T):
    rng = np.random.default_rng(T)
    B, V = 512, 5
    parent, cand, top = _random_accept_case(rng, B, T, V)
    prefix = rng.integers(0, 300, size=B).astype(np.int32)
    S_max = 300 + T // 2                 # some sequences overflow the cache
    ref = oracle.accept_path(top, cand, parent, prefix, V, S_max)
    d = lambda a: i32(a, cuda_device)
    outs = {k: torch.full((B,), -9, dtype=torch.int32, device=cuda_device)
            for k in ("accept_len", "next_token", "new_prefix_len", "status")}
    path = torch.full((B, T), -9, dtype=torch.int32, device=cuda_device)
    ppd.ppd_accept_path(d(top), d(cand), d(parent), d(prefix), V, S_max, outs["accept_len"], path,
                        outs["next_token"], outs["new_prefix_len"], outs["status"])
    torch.cuda.synchronize()
    for k in ("accept_len", "next_token", "new_prefix_len", "status"):
        np.testing.assert_array_equal(outs[k].cpu().numpy(), ref[k], err_msg=k)
    np.testing.assert_array_equal(path.cpu().numpy(), ref["path"])


def test_accept_path_errors(cuda_device):
    parent = np.array([[-1, 0, 1], [-1, 2, 0], [0, 0, 1], [-1, 0, 1], [-1, 0, 1]], np.int32)
    cand = np.array([[1, 2, 3], [1, 2, 3], [1, 2, 3], [1, 9, 3], [-1, 2, 3]], np.int32)
    top = np.array([[2, 3, 0]] * 5, np.int32)
    prefix = np.array([5, 5, 5, 5, 5], np.int32)
    ref = oracle.accept_path(top, cand, parent, prefix, 8, 100)
    B, T = parent.shape
    d = lambda a: i32(a, cuda_device)
    o = [torch.empty(B, dtype=torch.int32, device=cuda_device) for _ in range(4)]
    path = torch.empty((B, T), dtype=torch.int32, device=cuda_device)
    ppd.ppd_accept_path(d(top), d(cand), d(parent), d(prefix), 8, 100, o[0], path, o[1], o[2], o[3])
    torch.cuda.synchronize()
    assert o[3].cpu().tolist() == ref["status"].tolist() == [0, 3, 3, 3, 3]
    assert o[0].cpu().tolist() == ref["accept_len"].tolist()
    np.testing.assert_array_equal(path.cpu().numpy(), ref["path"])


# ----------------------------------------------------------------------------- compaction

@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_kv_compact_matches_oracle(cuda_device, dtype):
    rng = np.random.default_rng(3)
    L, B, H, T, D, S = 3, 4, 5, 64, 128, 400
    g = torch.Generator().manual_seed(0)
    mk = lambda *s: torch.randn(s, generator=g).to(dtype)
    kc, vc, kt, vt = mk(L, B, H, S, D), mk(L, B, H, S, D), mk(L, B, H, T, D), mk(L, B, H, T, D)
    acc = np.array([7, 1, 0, 3], np.int32)
    pre = np.array([10, 399, 50, 200], np.int32)
    path = np.full((B, T), -1, np.int32)
    for b in range(B):
        path[b, :acc[b]] = np.sort(rng.choice(T, acc[b], replace=False))
    ek, ev = oracle.kv_compact(kc, vc, kt, vt, path, acc, pre)
    dk, dv = kc.to(cuda_device), vc.to(cuda_device)
    ppd.ppd_kv_compact(dk, dv, kt.to(cuda_device), vt.to(cuda_device), i32(path, cuda_device),
                       i32(acc, cuda_device), i32(pre, cuda_device))
    torch.cuda.synchronize()
    view, npv = (torch.int16, np.int16) if dtype == torch.bfloat16 else (torch.int32, np.int32)
    np.testing.assert_array_equal(dk.cpu().view(view).numpy(), ek.view(npv))
    np.testing.assert_array_equal(dv.cpu().view(view).numpy(), ev.view(npv))


# ----------------------------------------------------------------------------- full step

def _verify_step(w, s, t, dev, units=None):
    g = {k: v.to(dev) for k, v in t.items()}
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev, with_lse=True)
    ppd.ppd_verify_step(g["q"], g["k_cache"], g["v_cache"], g["k_tree"], g["v_tree"],
                        i32(s.prefix_len, dev), i32(s.parent, dev), i32(s.cand_tokens, dev),
                        torch.from_numpy(s.logits).to(dev), bufs.out, bufs.argmax, bufs.accept_len,
                        bufs.path, bufs.next_token, bufs.new_prefix_len, bufs.dev_status,
                        bufs.workspace, lse=bufs.lse)
    torch.cuda.synchronize()
    return g, bufs


@pytest.mark.parametrize("name,overrides", [("tiny", {}), ("tiny", {"B": 4}),
                                            ("mobilellama", {"L": 2, "H": 4}),
                                            ("vicuna7b", {"L": 1, "H": 2, "B": 2}),
                                            ("mobilellama", {"L": 1, "H": 2, "B": 2, "T": 285,
                                                             "n_cand": 72})])
def test_verify_step_matches_oracle(cuda_device, name, overrides):
    w = W.scaled(W.WORKLOADS[name], **overrides)
    s = W.make_step_inputs(w)
    t = tensors(w, prefix_len=s.prefix_len)
    g, bufs = _verify_step(w, s, t, cuda_device)
    ref = oracle.verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                             s.prefix_len, s.parent, s.cand_tokens, s.logits)
    assert_attn_close(bufs.out.cpu().numpy().reshape(ref["out"].shape), ref["out"], name)
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), ref["argmax"])
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), ref["status"])
    assert (ref["accept_len"] >= 1).all()
    np.testing.assert_array_equal(g["k_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["k_cache"])
    np.testing.assert_array_equal(g["v_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["v_cache"])


def test_verify_step_is_repeatable(cuda_device):
    """Running the same step twice gives identical outputs (compaction reads the
    tree buffers, never the rows it writes)."""
    w = W.scaled(W.WORKLOADS["mobilellama"], L=2, H=4)
    s = W.make_step_inputs(w)
    t = tensors(w)
    g, b1 = _verify_step(w, s, t, cuda_device)
    out1 = b1.out.clone()
    kc1 = g["k_cache"].clone()
    g2, b2 = _verify_step(w, s, t, cuda_device)
    assert torch.equal(out1, b2.out)
    assert torch.equal(kc1.view(torch.int16), g2["k_cache"].view(torch.int16))


@pytest.mark.parametrize("B", [64, 65])
def test_verify_step_batch_paths(cuda_device, B):
    """B <= 64 runs the fused step (here with an argmax grid first: the logits
    outweigh the short prefixes); larger batches run separate grids."""
    w = W.Workload("batch", L=1, B=B, H=2, D=64, P=40, T=16, V=300, n_cand=8, max_depth=3,
                   chains="every1", match_rate=0.8, seed=B)
    rng = np.random.default_rng(B)
    pl = rng.integers(0, 41, size=B).astype(np.int32)
    s = W.make_step_inputs(w, prefix_len=pl)
    t = tensors(w, prefix_len=pl)
    g, bufs = _verify_step(w, s, t, cuda_device)
    ref = oracle.verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                             s.prefix_len, s.parent, s.cand_tokens, s.logits)
    assert_attn_close(bufs.out.cpu().numpy().reshape(ref["out"].shape), ref["out"], f"B={B}")
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), ref["argmax"])
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), ref["status"])
    np.testing.assert_array_equal(g["k_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["k_cache"])
    np.testing.assert_array_equal(g["v_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["v_cache"])


def test_verify_step_reports_bad_sequences(cuda_device):
    """Per-sequence device status in the fused step: a malformed tree and a
    path that does not fit leave those sequences unaccepted and uncompacted."""
    w = W.scaled(W.WORKLOADS["tiny"], B=3)
    s = W.make_step_inputs(w)
    s.parent[1, 7] = 9                       # parent after child
    s.prefix_len[2] = w.S_max                # no room for even the root
    t = tensors(w, prefix_len=s.prefix_len)
    g, bufs = _verify_step(w, s, t, cuda_device)
    ref = oracle.verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                             s.prefix_len, s.parent, s.cand_tokens, s.logits)
    assert bufs.dev_status.cpu().tolist() == ref["status"].tolist() == [0, 3, 4]
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    np.testing.assert_array_equal(g["k_cache"].cpu().view(torch.int16).numpy().view(np.uint16),
                                  ref["k_cache"])
