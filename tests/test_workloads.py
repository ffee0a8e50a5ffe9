"""Seeded input generators: determinism and the tree / logit properties that
the paper's customised sparse tree (Section 4.1) and the workload recipes
require."""
import numpy as np
import pytest

from paper_2405_18628_gb300 import workloads as W


def _depths(parent):
    d = np.zeros(len(parent), int)
    for i in range(1, len(parent)):
        d[i] = d[parent[i]] + 1
    return d


@pytest.mark.parametrize("name", ["tiny", "mobilellama", "vicuna7b", "vicuna13b",
                                  "sweep_t16", "sweep_t128"])
def test_tree_shape(name):
    w = W.WORKLOADS[name]
    rng = np.random.Generator(np.random.PCG64(w.seed))
    for _ in range(20):
        parent, is_prompt = W.make_tree(rng, w)
        assert parent.shape == (w.T,)
        assert parent[0] == -1
        assert all(0 <= parent[i] < i for i in range(1, w.T))
        assert (~is_prompt).sum() == w.n_cand
        assert not is_prompt[:w.n_cand].any() and is_prompt[w.n_cand:].all()
        d = _depths(parent)
        assert d[:w.n_cand].max() <= w.max_depth
        # a prompt node's parent is its anchor candidate or the previous prompt node
        for i in range(w.n_cand, w.T):
            p = parent[i]
            assert p < w.n_cand or p == i - 1
        if w.chains.startswith("every"):
            c = int(w.chains[5:])
            for a in range(w.n_cand):
                kids = [i for i in range(w.n_cand, w.T) if parent[i] == a]
                assert len(kids) == 1
                n, cur = 1, kids[0]
                while cur + 1 < w.T and parent[cur + 1] == cur:
                    n += 1
                    cur += 1
                assert n == c


def test_generator_deterministic():
    w = W.WORKLOADS["tiny"]
    a = W.make_step_inputs(w)
    b = W.make_step_inputs(w)
    for f in ("parent", "cand_tokens", "prefix_len", "logits", "top"):
        np.testing.assert_array_equal(getattr(a, f), getattr(b, f))
    c = W.make_step_inputs(w, seed=w.seed + 1)
    assert not np.array_equal(a.logits, c.logits)
    ta = W.make_tensors(w)
    tb = W.make_tensors(w)
    for k in ta:
        assert (ta[k].float() == tb[k].float()).all()


def test_planted_top_is_unique_max():
    rng = np.random.Generator(np.random.PCG64(7))
    logits, top = W.planted_logits(rng, 300, 1024)
    assert logits.dtype == np.float32
    np.testing.assert_array_equal(np.argmax(logits, axis=1), top)
    mx = logits.max(axis=1)
    assert ((logits == mx[:, None]).sum(axis=1) == 1).all()
    # marginal law: N(0,1) mean/var over all entries, max near the V-sample quantile
    assert abs(logits.mean()) < 0.01 and abs(logits.var() - 1.0) < 0.02
    from scipy.special import ndtri
    assert abs(np.median(mx) - ndtri(0.5 ** (1 / 1024))) < 0.1
    # top index uniform: chi-square over 8 bins
    counts = np.bincount(top * 8 // 1024, minlength=8)
    assert ((counts - 300 / 8) ** 2 / (300 / 8)).sum() < 30


def test_candidate_tokens_and_match_rate():
    w = W.scaled(W.WORKLOADS["vicuna7b"], B=64, V=512)
    s = W.make_step_inputs(w)
    prompt = s.cand_tokens == -1
    assert (prompt.sum(axis=1) == w.T - w.n_cand).all()
    assert ((s.cand_tokens[~prompt] >= 0) & (s.cand_tokens[~prompt] < w.V)).all()
    hits = []
    for b in range(w.B):
        for i in range(1, w.n_cand):
            hits.append(s.cand_tokens[b, i] == s.top[b, s.parent[b, i]])
    rate = np.mean(hits)
    expect = w.match_rate + (1 - w.match_rate) / w.V
    assert abs(rate - expect) < 4 * np.sqrt(expect * (1 - expect) / len(hits))


def test_poisoned_tail():
    w = W.WORKLOADS["tiny"]
    t = W.make_tensors(w, poison_tail=True)
    import torch
    assert torch.isnan(t["k_cache"][:, :, :, w.P:].float()).all()
    assert not torch.isnan(t["k_cache"][:, :, :, :w.P].float()).any()
