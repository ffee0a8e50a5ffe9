"""The fused verification step at the full workload sizes, in the launch
configuration the benchmark times.  Inputs are drawn on the device; the oracle
checks every index output in full and the attention outputs of every
(layer, sequence, head) slice for the MobileLlama- and Vicuna-7B-shaped
workloads, and of every sequence and head of the first, the last and four
seeded random layers for the larger ones (max-abs and relative L2 over all
outputs checked); compaction is checked row by row on the device against the
tree rows the path names."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ATOL, RTOL_L2 = 5e-3, 1e-3


def _row_checksums(x):
    """Per (l,b,h,row) int64 sums of the raw bit patterns, one layer at a time."""
    return torch.stack([x[l].view(torch.int16).to(torch.int64).sum(dim=-1)
                        for l in range(x.shape[0])])


@pytest.mark.parametrize("name", ["mobilellama", "vicuna7b", "vicuna13b",
                                  "sweep_t16", "sweep_t32", "sweep_t64", "sweep_t128"])
def test_full_size_step(cuda_device, name):
    w = W.WORKLOADS[name]
    need = 2 * w.L * w.B * w.H * (w.S_max + 2 * w.T) * w.D * 2
    torch.cuda.empty_cache()                    # earlier cases' blocks back to the device
    free, _ = torch.cuda.mem_get_info()
    if need * 1.3 > free:
        pytest.skip(f"{name} needs {need / 2**30:.0f} GiB")
    s = W.make_step_inputs(w)
    t = W.make_tensors(w, device=cuda_device)
    before = {k: _row_checksums(t[k]) for k in ("k_cache", "v_cache")}
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(cuda_device)
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=cuda_device)
    ppd.ppd_verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                        i32(s.prefix_len), i32(s.parent), i32(s.cand_tokens),
                        torch.from_numpy(s.logits).to(cuda_device), bufs.out, bufs.argmax,
                        bufs.accept_len, bufs.path, bufs.next_token, bufs.new_prefix_len,
                        bufs.dev_status, bufs.workspace)
    torch.cuda.synchronize()

    # indices: in full
    am = oracle.node_argmax(s.logits)
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), am)
    np.testing.assert_array_equal(am, s.top)                   # the planted maxima
    acc = oracle.accept_path(am, s.cand_tokens, s.parent, s.prefix_len, w.V, w.S_max)
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), acc[k], err_msg=k)
    assert (bufs.dev_status.cpu().numpy() == 0).all() and (acc["status"] == 0).all()

    # compaction: accepted rows hold the named tree rows; every other row unchanged
    for b in range(w.B):
        n, P = int(acc["accept_len"][b]), int(s.prefix_len[b])
        src = torch.from_numpy(acc["path"][b, :n].astype(np.int64)).to(cuda_device)
        for k, kt in (("k_cache", "k_tree"), ("v_cache", "v_tree")):
            got = t[k][:, b, :, P:P + n].view(torch.int16)
            want = t[kt][:, b, :, :][:, :, src].view(torch.int16)
            assert torch.equal(got, want), (k, b)
    for k in ("k_cache", "v_cache"):
        after = _row_checksums(t[k])
        mask = torch.ones_like(after, dtype=torch.bool)
        for b in range(w.B):
            n, P = int(acc["accept_len"][b]), int(s.prefix_len[b])
            mask[:, b, :, P:P + n] = False
        assert torch.equal(after[mask], before[k][mask]), k

    # attention: every slice of the checked layers, one layer at a time (the
    # cache's prefix rows are untouched by compaction, so the step's inputs)
    if name in ("mobilellama", "vicuna7b"):
        layers = list(range(w.L))
    else:
        rng = np.random.default_rng(w.seed)
        inner = rng.choice(np.arange(1, w.L - 1), size=4, replace=False).tolist()
        layers = sorted({0, w.L - 1, *inner})
    err, d2, r2 = 0.0, 0.0, 0.0
    for l in layers:
        sl = lambda x: x[l:l + 1].cpu()
        ref, _, _, st = oracle.tree_attention(sl(t["q"]), sl(t["k_cache"]), sl(t["v_cache"]),
                                              sl(t["k_tree"]), sl(t["v_tree"]), s.prefix_len,
                                              s.parent)
        assert (st == 0).all()
        got = bufs.out[l].double().cpu().numpy().reshape(ref.shape)
        assert np.isfinite(got).all(), l
        err = max(err, float(np.abs(got - ref).max()))
        d2 += float(np.sum((got - ref) ** 2))
        r2 += float(np.sum(ref ** 2))
    rel = np.sqrt(d2 / r2)
    assert err <= ATOL and rel <= RTOL_L2, (layers, err, rel)


def _plant_ties(logits, chunk, r0=0):
    """Rows r0.. of one sequence's logits rewritten with ties, NaNs,
    infinities and signed zeros, many of them straddling the boundaries of the
    argmax's per-row column spans (columns k*chunk - 1 | k*chunk)."""
    logits = logits[r0:]
    T, V = logits.shape
    n_b = max(1, (V - 1) // chunk)
    for r in range(min(T, 7)):                           # max tied across a boundary
        k = 1 + r % n_b
        m = logits[r].max() + 1.0
        logits[r, [k * chunk, k * chunk - 1]] = m
    for r in range(7, min(T, 14)):                       # two NaNs either side of a boundary
        k = 1 + r % n_b
        logits[r, [k * chunk, k * chunk - 1]] = np.nan
    for r in range(14, min(T, 21)):                      # +inf in two chunks
        k = 1 + r % n_b
        logits[r, [k * chunk + 3, (k - 1) * chunk + 1]] = np.inf
    if T > 21:
        logits[21, :] = -np.inf                          # all equal: index 0
    if T > 22:
        logits[22, :] = -2.0
        logits[22, [chunk, chunk - 1]] = [0.0, -0.0]     # -0 == +0
    if T > 23:
        logits[23, V - 1] = np.nan                       # the only NaN, last column
    if T > 24:
        m = logits[24].max() + 0.5
        logits[24, [V - 1, 2 * chunk, chunk]] = m        # three-way tie


@pytest.mark.parametrize("name", ["mobilellama", "vicuna7b"])
def test_full_size_step_argmax_ties(cuda_device, name):
    """The fused step at full size, in the form the benchmark times, with ties,
    NaNs, +-inf and signed zeros planted across the column chunks of both
    in-grid argmax forms (the side warps' chunks of 4000 logits, rows 0..24;
    the softmax warps' chunks of 1000, rows 25..49): every index output and
    the compacted cache rows bit for bit against the oracle."""
    w = W.WORKLOADS[name]
    assert ppd.ppd_verify_step_form(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max) in (1, 2, 3)
    s = W.make_step_inputs(w)
    lg = s.logits.copy()
    for b in range(w.B):
        _plant_ties(lg[b], 4000)
        _plant_ties(lg[b], 1000, r0=25)
    am = oracle.node_argmax(lg)
    # candidates that copied their parent's planted top token now copy the new argmax
    cand = s.cand_tokens.copy()
    for b in range(w.B):
        for i in range(1, w.T):
            pa = s.parent[b, i]
            if cand[b, i] >= 0 and cand[b, i] == s.top[b, pa]:
                cand[b, i] = am[b, pa]
    t = W.make_tensors(w, device=cuda_device)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.int32)).to(cuda_device)
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=cuda_device)
    ppd.ppd_verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                        i32(s.prefix_len), i32(s.parent), i32(cand),
                        torch.from_numpy(lg).to(cuda_device), bufs.out, bufs.argmax,
                        bufs.accept_len, bufs.path, bufs.next_token, bufs.new_prefix_len,
                        bufs.dev_status, bufs.workspace)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), am)
    acc = oracle.accept_path(am, cand, s.parent, s.prefix_len, w.V, w.S_max)
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), acc[k], err_msg=k)
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), acc["status"])
    assert (acc["accept_len"] > 1).any()          # the rewritten rows still accept paths
    for b in range(w.B):
        n, P = int(acc["accept_len"][b]), int(s.prefix_len[b])
        src = torch.from_numpy(acc["path"][b, :n].astype(np.int64)).to(cuda_device)
        for k, kt in (("k_cache", "k_tree"), ("v_cache", "v_tree")):
            got = t[k][:, b, :, P:P + n].view(torch.int16)
            want = t[kt][:, b, :, :][:, :, src].view(torch.int16)
            assert torch.equal(got, want), (k, b)
