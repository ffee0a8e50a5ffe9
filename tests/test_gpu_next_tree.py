"""Next-step candidate tree on the GPU (through the C ABI) against the oracle,
bit for bit: the state k picked from the accepted node's prompt chains, the
top-K guesses per chain position (including ties, NaNs and -inf logits) over
one chain, the fp32 average of n_ept ensemble chains' logits or the mean of
their probabilities (near-ties of the latter within fp32 rounding), and the assembled
parent / candidate arrays; bad templates and failed sequences report
PPD_ERR_TREE."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

from test_gpu_parity import i32
from test_oracle_next_tree import _softmax_rows

pytestmark = pytest.mark.gpu


def _run(dev, logits, parent, cand, path, accept_len, next_token, tp, tr, K, n_ept=1,
         ept_mean="logits"):
    B, T = parent.shape
    n_states, T_next = tp.shape
    out = {"next_parent": torch.full((B, T_next), -9, dtype=torch.int32, device=dev),
           "next_cand": torch.full((B, T_next), -9, dtype=torch.int32, device=dev),
           "next_state": torch.full((B,), -9, dtype=torch.int32, device=dev),
           "status": torch.full((B,), -9, dtype=torch.int32, device=dev)}
    ppd.ppd_next_tree(torch.from_numpy(np.ascontiguousarray(logits)).to(dev), i32(parent, dev),
                      i32(cand, dev), i32(path, dev), i32(accept_len, dev), i32(next_token, dev),
                      i32(tp, dev), i32(tr, dev), K, out["next_parent"], out["next_cand"],
                      out["next_state"], out["status"], n_ept=n_ept, ept_mean=ept_mean)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _compare(got, ref):
    for k in ("next_parent", "next_cand", "next_state", "status"):
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)


@pytest.mark.parametrize("name,overrides,n_states,T_next,K", [
    ("tiny", {"B": 6}, 4, 48, 4),
    ("mobilellama", {}, 5, 64, 8),
    ("vicuna7b", {"B": 3}, 4, 96, 16),
    ("sweep_t32", {"B": 8}, 3, 32, 1),
])
def test_next_tree_matches_oracle(cuda_device, name, overrides, n_states, T_next, K):
    w = W.scaled(W.WORKLOADS[name], **overrides)
    s = W.make_step_inputs(w)
    logits = s.logits.copy()
    logits[0, :, 5] = logits[0, :, 7] = 40.0          # ties at the top of every row of sequence 0
    if w.B > 1:
        logits[1, :, 11] = np.nan                     # NaN ranks first
        logits[1, :, :3] = -np.inf
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    tp, tr = W.make_tree_templates(n_states, T_next, K, np.random.default_rng(w.T + K))
    ref = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                           acc["next_token"], tp, tr, K)
    assert (ref["status"] == 0).all()
    got = _run(cuda_device, logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
               acc["next_token"], tp, tr, K)
    _compare(got, ref)


def test_next_tree_every_state(cuda_device):
    """Hand-built trees whose accepted node carries prompt chains of length 0..5:
    every state (capped at n_states - 1) is taken."""
    B, T, V, K = 6, 12, 300, 3
    parent = np.zeros((B, T), np.int32)
    cand = np.zeros((B, T), np.int32)
    path = np.full((B, T), -1, np.int32)
    for b in range(B):
        # root 0 -> candidate 1; chain of b prompt tokens under 1; the rest prompt nodes under 0
        parent[b] = [-1, 0] + [1 + j for j in range(b)] + [0] * (T - 2 - b)
        parent[b, 2] = 1 if b >= 1 else 0
        cand[b] = [3, 4] + [-1] * (T - 2)
        path[b, :2] = [0, 1]
    rng = np.random.default_rng(9)
    logits = rng.standard_normal((B, T, V)).astype(np.float32)
    accept_len = np.full(B, 2, np.int32)
    next_token = np.arange(B, dtype=np.int32) + 10
    tp, tr = W.make_tree_templates(4, 40, K, rng)
    ref = oracle.next_tree(logits, parent, cand, path, accept_len, next_token, tp, tr, K)
    assert ref["next_state"].tolist() == [0, 1, 2, 3, 3, 3]
    got = _run(cuda_device, logits, parent, cand, path, accept_len, next_token, tp, tr, K)
    _compare(got, ref)


def test_next_tree_errors(cuda_device):
    B, T, V, K = 3, 4, 50, 2
    parent = np.array([[-1, 0, 1, 2]] * B, np.int32)
    cand = np.array([[3, -1, -1, -1]] * B, np.int32)
    path = np.array([[0, -1, -1, -1]] * B, np.int32)
    logits = np.random.default_rng(1).standard_normal((B, T, V)).astype(np.float32)
    tp = np.array([[-1, 0, 1], [-1, 0, 0], [-1, 0, 1]], np.int32)
    tr = np.array([[0, -1, -1], [0, 0, 1], [0, 0, 3]], np.int32)   # state 2: rank 3 >= K
    accept_len = np.array([1, 0, 1], np.int32)                      # sequence 1 failed
    next_token = np.array([5, 5, -1], np.int32)                     # sequence 2: no next token
    ref = oracle.next_tree(logits, parent, cand, path, accept_len, next_token, tp, tr, K)
    got = _run(cuda_device, logits, parent, cand, path, accept_len, next_token, tp, tr, K)
    _compare(got, ref)
    assert got["status"].tolist() == [3, 3, 3]       # state 2 template bad; failed; no token


@pytest.mark.parametrize("n_ept,c,T_next,K", [(2, 3, 64, 8), (3, 2, 96, 16), (5, 1, 48, 4),
                                           (4, 3, 128, 16)])
def test_next_tree_ensemble_tokens(cuda_device, n_ept, c, T_next, K):
    """n_ept ensemble chains on every candidate (Section 3, Ensemble Prompt
    Tokens): guesses from the chains' averaged logits, state from the
    shortest chain; NaN and -inf logits included."""
    w = W.scaled(W.WORKLOADS["mobilellama"], B=6, T=16 * (1 + n_ept * c), n_cand=16,
                 chains=f"ept{n_ept}x{c}")
    s = W.make_step_inputs(w, seed=n_ept * 10 + c)
    logits = s.logits.copy()
    logits[0, :, 17] = np.nan
    logits[1, :, :9] = -np.inf
    logits[2, :, 100] = np.inf                    # +inf + -inf averages to NaN
    logits[2, ::2, 101] = -np.inf
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    tp, tr = W.make_tree_templates(c + 2, T_next, K, np.random.default_rng(K), n_ept=n_ept)
    for ne in (n_ept, 1, n_ept + 1):              # n_ept + 1: too few heads, state 0
        ref = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                               acc["next_token"], tp, tr, K, n_ept=ne)
        got = _run(cuda_device, logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                   acc["next_token"], tp, tr, K, n_ept=ne)
        _compare(got, ref)
        if ne == n_ept + 1:
            assert (got["next_state"][got["status"] == 0] == 0).all()
        elif ne == n_ept:
            assert (got["next_state"][got["status"] == 0] == min(c, c + 1)).all()


def test_next_tree_ensemble_hand_tree(cuda_device):
    """Two chains under the accepted node whose averaged logits rank
    differently from either chain alone (the oracle's hand-worked case)."""
    parent = np.array([[-1, 0, 1, 1, 2, 3, 0]] * 2, np.int32)
    parent[1, 5] = 0                              # sequence 1: chain 2 one position short
    cand = np.array([[9, 4, -1, -1, -1, -1, -1]] * 2, np.int32)
    logits = np.zeros((2, 7, 4), np.float32)
    logits[:, 2] = [4, 0, 1, 0]
    logits[:, 3] = [0, 6, 1, 0]
    logits[:, 4] = [1, 5, 0, 2]
    logits[:, 5] = [3, -5, 0, 2]
    path = np.array([[0, 1, -1, -1, -1, -1, -1]] * 2, np.int32)
    tp = np.array([[-1, 0, 1, 2, 3], [-1, 0, 0, 1, 2], [-1, 0, 1, 1, 0]], np.int32)
    tr = np.array([[0, -1, -1, -1, -1], [0, 0, -1, -1, -1], [0, 0, 0, 1, -1]], np.int32)
    alen, nt = np.array([2, 2], np.int32), np.array([7, 8], np.int32)
    got = _run(cuda_device, logits, parent, cand, path, alen, nt, tp, tr, 2, n_ept=2)
    assert got["status"].tolist() == [0, 0] and got["next_state"].tolist() == [2, 1]
    assert got["next_cand"].tolist() == [[7, 1, 0, 3, -1], [8, 1, -1, -1, -1]]
    ref = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, 2, n_ept=2)
    _compare(got, ref)


def test_next_tree_probability_mean_hand_tree(cuda_device):
    """The hand-worked tree with the chains' probabilities averaged (Section 3,
    Ensemble Prompt Tokens): position 2 ranks 1, 0 where the logit average
    ranks 0, 3."""
    parent = np.array([[-1, 0, 1, 1, 2, 3, 0]] * 2, np.int32)
    parent[1, 5] = 0
    cand = np.array([[9, 4, -1, -1, -1, -1, -1]] * 2, np.int32)
    logits = np.zeros((2, 7, 4), np.float32)
    logits[:, 2] = [4, 0, 1, 0]
    logits[:, 3] = [0, 6, 1, 0]
    logits[:, 4] = [1, 5, 0, 2]
    logits[:, 5] = [3, -5, 0, 2]
    path = np.array([[0, 1, -1, -1, -1, -1, -1]] * 2, np.int32)
    tp = np.array([[-1, 0, 1, 2, 3], [-1, 0, 0, 1, 2], [-1, 0, 1, 1, 0]], np.int32)
    tr = np.array([[0, -1, -1, -1, -1], [0, 0, -1, -1, -1], [0, 0, 0, 1, -1]], np.int32)
    alen, nt = np.array([2, 2], np.int32), np.array([7, 8], np.int32)
    got = _run(cuda_device, logits, parent, cand, path, alen, nt, tp, tr, 2, n_ept=2,
               ept_mean="probs")
    assert got["status"].tolist() == [0, 0] and got["next_state"].tolist() == [2, 1]
    assert got["next_cand"].tolist() == [[7, 1, 1, 0, -1], [8, 1, -1, -1, -1]]
    ref = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, 2, n_ept=2,
                           ept_mean="probs")
    _compare(got, ref)


def _chains(parent, cand, path, accept_len, b, n_ept):
    """The n_ept prompt chains below sequence b's accepted node, as node lists."""
    T = parent.shape[1]
    e = path[b, accept_len[b] - 1]
    kids = lambda u: [i for i in range(T) if parent[b, i] == u and cand[b, i] == -1]
    chains = []
    for head in kids(e)[:n_ept]:
        chain = [head]
        while kids(chain[-1]):
            chain.append(kids(chain[-1])[0])
        chains.append(chain)
    return chains


def _compare_probs(got, ref, logits, parent, cand, path, accept_len, tp, tr, n_ept):
    """Exact on state, status and parents; a guess may differ from the oracle's
    only where the two tokens' fp64 mean probabilities agree to 1e-4 relative
    (the kernel ranks fp32 sums: each chain's log-sum-exp carries up to ~1e-5
    relative error, which reweights the chains)."""
    for k in ("next_parent", "next_state", "status"):
        np.testing.assert_array_equal(got[k], ref[k], err_msg=k)
    n_diff = 0
    for b in np.nonzero(ref["status"] == 0)[0]:
        k = ref["next_state"][b]
        if k == 0:
            np.testing.assert_array_equal(got["next_cand"][b], ref["next_cand"][b])
            continue
        chains = _chains(parent, cand, path, accept_len, b, n_ept)
        with np.errstate(invalid="ignore", over="ignore"):
            pbar = [np.mean([_softmax_rows(logits[b, c[d]][None])[0] for c in chains], 0)
                    for d in range(k)]
        for i in range(tp.shape[1]):
            g, r = got["next_cand"][b, i], ref["next_cand"][b, i]
            if i == 0 or tr[k, i] < 0 or g == r:
                assert g == r, (b, i)
                continue
            depth, a = 0, i
            while a > 0:
                depth, a = depth + 1, tp[k, a]
            pg, pr = pbar[depth - 1][g], pbar[depth - 1][r]
            assert not np.isnan(pr) and abs(pg - pr) <= 1e-4 * pr, (b, i, g, r, pg, pr)
            n_diff += 1
    return n_diff


@pytest.mark.parametrize("n_ept,c,T_next,K", [(2, 3, 64, 8), (3, 2, 96, 16), (4, 3, 128, 16)])
def test_next_tree_probability_mean(cuda_device, n_ept, c, T_next, K):
    """The probability-mean guesses at MobileLlama's vocabulary against the
    oracle's fp64 ones; a NaN, a +inf and an all -inf row each turn a chain's
    probabilities into NaN, so that sequence's guesses fall back to index order
    exactly as in the oracle; -inf entries have probability 0."""
    w = W.scaled(W.WORKLOADS["mobilellama"], B=6, T=16 * (1 + n_ept * c), n_cand=16,
                 chains=f"ept{n_ept}x{c}")
    s = W.make_step_inputs(w, seed=n_ept * 10 + c + 1)
    logits = s.logits.copy() * 3.0                # sharper rows: a wide probability range
    logits[0, :, 17] = np.nan
    logits[1, :, :9] = -np.inf
    logits[2, :, 100] = np.inf
    logits[3, 1::3] = -np.inf                     # whole rows: no finite entry
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    tp, tr = W.make_tree_templates(c + 2, T_next, K, np.random.default_rng(K + 1), n_ept=n_ept)
    for ne in (n_ept, 1, n_ept + 1):
        ref = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                               acc["next_token"], tp, tr, K, n_ept=ne, ept_mean="probs")
        got = _run(cuda_device, logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                   acc["next_token"], tp, tr, K, n_ept=ne, ept_mean="probs")
        if ne == n_ept:
            assert (ref["status"] == 0).sum() >= 4
            n_diff = _compare_probs(got, ref, logits, s.parent, s.cand_tokens, acc["path"],
                                    acc["accept_len"], tp, tr, ne)
            assert n_diff <= 2
        else:
            _compare(got, ref)


@pytest.mark.parametrize("ept_mean", ["logits", "probs"])
def test_next_tree_128_ensemble_chains(cuda_device, ept_mean):
    """The largest ensemble the API takes: 128 prompt chains of two tokens
    under the accepted candidate (nodes 2..129 the heads, 130..257 their
    children), K = 16 guesses per depth; every chain's block of warps runs."""
    n_ept, T, V, K = 128, 258, 1000, 16
    parent = np.zeros((1, T), np.int32)
    parent[0, 0] = -1
    parent[0, 1] = 0
    parent[0, 2:130] = 1
    parent[0, 130:258] = np.arange(2, 130)
    cand = np.full((1, T), -1, np.int32)
    cand[0, :2] = [5, 6]
    path = np.full((1, T), -1, np.int32)
    path[0, :2] = [0, 1]
    rng = np.random.default_rng(128)
    logits = (2.0 * rng.standard_normal((1, T, V))).astype(np.float32)
    alen, nt = np.array([2], np.int32), np.array([9], np.int32)
    tp, tr = W.make_tree_templates(3, 40, K, rng)
    ref = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K, n_ept=n_ept,
                           ept_mean=ept_mean)
    assert ref["status"].tolist() == [0] and ref["next_state"].tolist() == [2]
    got = _run(cuda_device, logits, parent, cand, path, alen, nt, tp, tr, K, n_ept=n_ept,
               ept_mean=ept_mean)
    if ept_mean == "logits":
        _compare(got, ref)
    else:
        assert _compare_probs(got, ref, logits, parent, cand, path, alen, tp, tr, n_ept) <= 2


@pytest.mark.parametrize("V,K", [(40, 16), (37, 5), (300, 16)])
def test_next_tree_small_vocab_split_rows(cuda_device, V, K):
    """Vocabularies so small that each of the blocks sharing a row holds fewer
    columns than K (V = 40: ten blocks of four columns for sixteen guesses;
    V = 37: no 16-byte loads), with ties and NaNs: the merged guesses are
    still the oracle's, bit for bit, in both averaging modes."""
    w = W.scaled(W.WORKLOADS["tiny"], B=2, V=V, T=16 * (1 + 2 * 3), n_cand=16, chains="ept2x3")
    s = W.make_step_inputs(w, seed=V)
    logits = np.round(s.logits * 2.0).astype(np.float32)   # many ties
    logits[0, :, 3] = np.nan
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    tp, tr = W.make_tree_templates(4, 48, K, np.random.default_rng(V + K), n_ept=2)
    for ne, mode in ((2, "logits"), (1, "logits"), (2, "probs")):
        ref = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                               acc["next_token"], tp, tr, K, n_ept=ne, ept_mean=mode)
        got = _run(cuda_device, logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                   acc["next_token"], tp, tr, K, n_ept=ne, ept_mean=mode)
        if mode == "probs":
            assert _compare_probs(got, ref, logits, s.parent, s.cand_tokens, acc["path"],
                                  acc["accept_len"], tp, tr, ne) <= 4
        else:
            _compare(got, ref)
        assert (ref["next_state"] > 0).any()
