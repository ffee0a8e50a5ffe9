"""Pins for the oracle's next-step candidate generation (Section 3 step (1):
the prompt tokens appended to the accepted token predict the following
tokens; Section 3, Ensemble Prompt Tokens: n_ept tokens per prompt position,
the guess from the average of their logits; Appendix, Definition of tree
states: the next tree takes state T_k, whose candidate subtree is at most k
deep).

Expected values come from numpy's stable argsort (top-k order), hand-worked
examples (one and two ensemble chains), an independent restatement on small
random cases (chains found from per-node child lists, averages by an explicit
fp32 loop, ranks by numpy), and the state rule."""
import numpy as np
import pytest

import oracle
from paper_2405_18628_gb300 import workloads as W


def test_topk_matches_numpy_stable_sort():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal((7, 301)) * 2).astype(np.float32)
    x[0, [10, 20, 30]] = x[0].max() + 1.0          # a three-way tie at the top: lower index first
    x[1, :] = 0.0                                   # all equal: indices 0, 1, 2, ...
    got = oracle.topk(x, 9)
    for r in range(x.shape[0]):
        ref = np.lexsort((np.arange(x.shape[1]), -x[r]))[:9]
        assert got[r].tolist() == ref.tolist(), r
    assert got[0, :3].tolist() == [10, 20, 30]
    assert got[1].tolist() == list(range(9))


def test_topk_nan_first_then_values():
    x = np.array([[1.0, np.nan, 5.0, np.nan, 3.0, 5.0]], np.float32)
    assert oracle.topk(x, 6)[0].tolist() == [1, 3, 2, 5, 4, 0]
    # rank 0 is the argmax rule
    rng = np.random.default_rng(4)
    y = rng.standard_normal((20, 77)).astype(np.float32)
    assert (oracle.topk(y, 1)[:, 0] == oracle.node_argmax(y)).all()


def test_hand_worked_example():
    # this step's tree: 0 root; 1, 2 candidates under 0; 3 candidate under 1;
    # 4 -> 5 -> 6 a prompt chain under 3; 7 a prompt node under 2.
    parent = np.array([[-1, 0, 0, 1, 3, 4, 5, 2]])
    cand = np.array([[9, 4, 7, 2, -1, -1, -1, -1]])
    V = 6
    logits = np.zeros((1, 8, V), np.float32)
    logits[0, 4] = [0, 1, 5, 3, 2, 4]      # chain node c_1 -> ranking 2, 5, 3, 4, 1, 0
    logits[0, 5] = [6, 0, 0, 7, 0, 1]      # c_2 -> 3, 0, 5, 1, 2, 4
    logits[0, 6] = [9, 9, 9, 9, 9, 9]      # c_3 -> 0, 1, 2, ...
    path = np.array([[0, 1, 3, -1, -1, -1, -1, -1]])
    accept_len, next_token = np.array([3]), np.array([4])
    # templates for states 0..2 with T_next = 6
    tp = np.array([[-1, 0, 1, 2, 3, 4],            # k=0: root + a prompt chain
                   [-1, 0, 0, 1, 2, 3],            # k=1: two depth-1 candidates (ranks 1, 0)
                   [-1, 0, 1, 1, 0, 4]])           # k=2: depth1 r0, depth2 r0 and r2, prompts
    tr = np.array([[0, -1, -1, -1, -1, -1],
                   [0, 1, 0, -1, -1, -1],
                   [0, 0, 0, 2, -1, -1]])
    r = oracle.next_tree(logits, parent, cand, path, accept_len, next_token, tp, tr, K=3)
    # end node 3 has the chain 4, 5, 6 (k = 3), capped at n_states - 1 = 2
    assert r["status"].tolist() == [0] and r["next_state"].tolist() == [2]
    assert r["next_parent"][0].tolist() == [-1, 0, 1, 1, 0, 4]
    # node 1: depth 1 rank 0 -> c_1's best (2); nodes 2, 3: depth 2 ranks 0, 2 -> c_2's 3 and 5
    assert r["next_cand"][0].tolist() == [4, 2, 3, 5, -1, -1]


def _softmax_rows(x):
    """fp64 softmax of each row, written out: a row holding a NaN, or whose
    largest entry is +inf or -inf, gives NaN everywhere (numpy's inf - inf)."""
    x = np.asarray(x, np.float64)
    m = np.where(np.isnan(x).any(-1), np.nan, np.max(np.where(np.isnan(x), -np.inf, x), -1))
    with np.errstate(invalid="ignore"):
        lse = m + np.log(np.exp(x - m[..., None]).sum(-1))
        return np.exp(x - lse[..., None])


def _independent(logits, parent, cand, path, accept_len, next_token, tp, tr, K, n_ept=1,
                 ept_mean="logits"):
    """Restatement: per-node lists of prompt children (lowest index first); the
    end node's first n_ept prompt children head the chains, each continued
    through first children; the average over the chains is an explicit fp32
    loop over logits, or (ept_mean="probs", n_ept > 1) the fp64 mean of the
    chains' softmax rows; ranks come from numpy."""
    B, T = parent.shape
    n_states, T_next = tp.shape
    out_p = np.full((B, T_next), -1)
    out_c = np.full((B, T_next), -1)
    out_s = np.full(B, -1)
    for b in range(B):
        e = path[b, accept_len[b] - 1]
        children = {u: sorted(i for i in range(T) if parent[b, i] == u and cand[b, i] == -1)
                    for u in range(T)}
        chains = []
        for head in children[e][:n_ept]:
            chain, u = [head], head
            while children[u]:
                u = children[u][0]
                chain.append(u)
            chains.append(chain)
        k = min(len(c) for c in chains) if len(chains) == n_ept else 0
        k = min(k, n_states - 1)
        ranks = []
        for d in range(k):
            if ept_mean == "probs" and n_ept > 1:
                avg = _softmax_rows(np.stack([logits[b, c[d]] for c in chains])).mean(0)
            else:
                acc = np.array(logits[b, chains[0][d]], np.float32)
                for c in chains[1:]:
                    acc = (acc + logits[b, c[d]]).astype(np.float32)
                avg = (acc / np.float32(n_ept)).astype(np.float32)
            nan = np.isnan(avg)          # NaN ranks first; numpy would sort it last
            ranks.append(np.lexsort((np.arange(logits.shape[2]), -np.where(nan, 0, avg), ~nan))[:K])
        depth = {0: 0}
        for i in range(1, T_next):
            depth[i] = depth[tp[k, i]] + 1 if tr[k, i] >= 0 else None
        out_p[b] = tp[k]
        out_c[b, 0] = next_token[b]
        for i in range(1, T_next):
            if tr[k, i] >= 0:
                out_c[b, i] = ranks[depth[i] - 1][tr[k, i]]
        out_s[b] = k
    return out_p, out_c, out_s


@pytest.mark.parametrize("seed", range(6))
def test_random_cases_match_independent_restatement(seed):
    rng = np.random.default_rng(seed)
    w = W.scaled(W.WORKLOADS["tiny"], B=5, V=200)
    s = W.make_step_inputs(w, seed=seed)
    acc = oracle.accept_path(oracle.node_argmax(s.logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    n_states, T_next, K = 3 + seed % 3, 24 + 8 * (seed % 2), 4
    tp, tr = W.make_tree_templates(n_states, T_next, K, rng)
    r = oracle.next_tree(s.logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                         acc["next_token"], tp, tr, K)
    ref_p, ref_c, ref_s = _independent(s.logits, s.parent, s.cand_tokens, acc["path"],
                                       acc["accept_len"], acc["next_token"], tp, tr, K)
    assert (r["status"] == 0).all()
    np.testing.assert_array_equal(r["next_parent"], ref_p)
    np.testing.assert_array_equal(r["next_cand"], ref_c)
    np.testing.assert_array_equal(r["next_state"], ref_s)


def _ept_hand_tree():
    """0 root; 1 candidate under 0; prompt nodes 2, 3 under 1 (two ensemble
    chains), 4 under 2 and 5 under 3 (their second positions), 6 under 0."""
    parent = np.array([[-1, 0, 1, 1, 2, 3, 0]])
    cand = np.array([[9, 4, -1, -1, -1, -1, -1]])
    logits = np.zeros((1, 7, 4), np.float32)
    logits[0, 2] = [4, 0, 1, 0]        # chain 1, position 1
    logits[0, 3] = [0, 6, 1, 0]        # chain 2, position 1 -> average [2, 3, 1, 0]
    logits[0, 4] = [1, 5, 0, 2]        # chain 1, position 2
    logits[0, 5] = [3, -5, 0, 2]       # chain 2, position 2 -> average [2, 0, 0, 2]
    logits[0, 6] = [0, 0, 0, 99]
    path = np.array([[0, 1, -1, -1, -1, -1, -1]])
    tp = np.array([[-1, 0, 1, 2, 3],
                   [-1, 0, 0, 1, 2],
                   [-1, 0, 1, 1, 0]])
    tr = np.array([[0, -1, -1, -1, -1],
                   [0, 0, -1, -1, -1],
                   [0, 0, 0, 1, -1]])     # state 2: depth 1 rank 0, depth 2 ranks 0 and 1
    return logits, parent, cand, path, np.array([2]), np.array([7]), tp, tr


def test_ept_hand_worked_example():
    logits, parent, cand, path, alen, nt, tp, tr = _ept_hand_tree()
    r = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2)
    # averaged rankings: position 1 -> 1, 0, 2, 3; position 2 -> 0, 3, 1, 2 (ties: lower index)
    assert r["status"].tolist() == [0] and r["next_state"].tolist() == [2]
    assert r["next_parent"][0].tolist() == [-1, 0, 1, 1, 0]
    assert r["next_cand"][0].tolist() == [7, 1, 0, 3, -1]
    # one ensemble token: chain 2 -> 4 alone, rankings 0, 2, ... and 1, 3, ...
    r1 = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=1)
    assert r1["next_cand"][0].tolist() == [7, 0, 1, 3, -1]
    assert (oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2)["next_cand"] ==
            r1["next_cand"]).all()
    # three ensemble tokens but only two prompt children: state 0
    r3 = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=3)
    assert r3["next_state"].tolist() == [0] and r3["next_cand"][0].tolist() == [7, -1, -1, -1, -1]


def test_ept_probability_mean_hand_worked_example():
    """The same tree with the chains' probabilities averaged (softmax by hand):
    position 1 -> mean [0.4615, 0.5026, 0.0262, 0.0097], ranking 1, 0, 2, 3;
    position 2 -> chain 1 softmax [0.0170, 0.9304, 0.0063, 0.0463], chain 2
    [0.7052, 0.0002, 0.0351, 0.2594], mean [0.3611, 0.4653, 0.0207, 0.1529],
    ranking 1, 0, 3, 2 -- where the logit average ranks 0, 3 first."""
    logits, parent, cand, path, alen, nt, tp, tr = _ept_hand_tree()
    r = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2,
                         ept_mean="probs")
    assert r["status"].tolist() == [0] and r["next_state"].tolist() == [2]
    assert r["next_parent"][0].tolist() == [-1, 0, 1, 1, 0]
    assert r["next_cand"][0].tolist() == [7, 1, 1, 0, -1]
    # one ensemble token: the probabilities rank as the logits do
    for n in (1, 3):
        rp = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=n,
                              ept_mean="probs")
        rl = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=n)
        for k in rp:
            np.testing.assert_array_equal(rp[k], rl[k], err_msg=k)
    with pytest.raises(ValueError):
        oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2,
                         ept_mean="mean")


def test_ept_probability_mean_is_shift_invariant():
    """Softmax ignores a constant added to a row: shifting one chain's logits by
    a large constant leaves the probability-mean guesses unchanged.  Averaging
    unnormalised exp(x) instead would let the shifted chain decide alone
    (guesses 7, 1, 0, 3)."""
    logits, parent, cand, path, alen, nt, tp, tr = _ept_hand_tree()
    a = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2,
                         ept_mean="probs")
    for c in (40.0, -60.0):
        shifted = logits.copy()
        shifted[0, [3, 5]] += c         # chain 2, both positions
        b = oracle.next_tree(shifted, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2,
                             ept_mean="probs")
        np.testing.assert_array_equal(a["next_cand"], b["next_cand"])


def test_ept_state_is_the_shortest_chain():
    logits, parent, cand, path, alen, nt, tp, tr = _ept_hand_tree()
    parent = parent.copy()
    parent[0, 5] = 0                   # chain 2 loses its second position
    r = oracle.next_tree(logits, parent, cand, path, alen, nt, tp, tr, K=2, n_ept=2)
    assert r["next_state"].tolist() == [1]
    assert r["next_cand"][0].tolist() == [7, 1, -1, -1, -1]
    assert r["next_parent"][0].tolist() == [-1, 0, 0, 1, 2]


@pytest.mark.parametrize("n_ept", [2, 4])
def test_ept_identical_chains_match_one_chain(n_ept):
    """With every ensemble chain carrying the same logits, the fp32 average of
    n_ept = 2^j copies is exact, so the guesses equal those of one chain."""
    rng = np.random.default_rng(n_ept)
    w = W.scaled(W.WORKLOADS["tiny"], B=3, V=300, T=16 * (1 + 2 * n_ept), chains=f"ept{n_ept}x2")
    s = W.make_step_inputs(w, seed=5)
    logits = s.logits.copy()
    for b in range(w.B):
        for i in range(w.T):
            if s.cand_tokens[b, i] == -1 and s.cand_tokens[b, s.parent[b, i]] != -1:
                # an ensemble head: copy the first sibling head's chain logits
                sib = [j for j in range(w.T) if s.parent[b, j] == s.parent[b, i]
                       and s.cand_tokens[b, j] == -1]
                first = sib[0]
                logits[b, i] = logits[b, first]
                ci = [j for j in range(w.T) if s.parent[b, j] == i]
                cf = [j for j in range(w.T) if s.parent[b, j] == first]
                logits[b, ci[0]] = logits[b, cf[0]]
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    tp, tr = W.make_tree_templates(3, 40, 4, rng, n_ept=n_ept)
    r = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                         acc["next_token"], tp, tr, 4, n_ept=n_ept)
    r1 = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                          acc["next_token"], tp, tr, 4, n_ept=1)
    # the probabilities of n_ept equal rows average (fp64, 2^j of them) to one row's
    rp = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                          acc["next_token"], tp, tr, 4, n_ept=n_ept, ept_mean="probs")
    assert (r["status"] == 0).all()
    for k in ("next_parent", "next_cand", "next_state"):
        np.testing.assert_array_equal(r[k], r1[k], err_msg=k)
        np.testing.assert_array_equal(rp[k], r1[k], err_msg=k)


@pytest.mark.parametrize("ept_mean", ["logits", "probs"])
@pytest.mark.parametrize("seed,n_ept", [(0, 2), (1, 3), (2, 2), (3, 5)])
def test_ept_random_cases_match_independent_restatement(seed, n_ept, ept_mean):
    rng = np.random.default_rng(100 + seed)
    c = 1 + seed % 3
    w = W.scaled(W.WORKLOADS["tiny"], B=4, V=257, T=12 * (1 + n_ept * c), n_cand=12,
                 chains=f"ept{n_ept}x{c}")
    s = W.make_step_inputs(w, seed=seed)
    logits = s.logits.copy()
    logits[0, :, 3] = np.nan
    logits[1, :, :5] = -np.inf
    acc = oracle.accept_path(oracle.node_argmax(logits), s.cand_tokens, s.parent, s.prefix_len,
                             w.V, w.S_max)
    n_states, K = 4, 5
    tp, tr = W.make_tree_templates(n_states, 48, K, rng, n_ept=n_ept)
    r = oracle.next_tree(logits, s.parent, s.cand_tokens, acc["path"], acc["accept_len"],
                         acc["next_token"], tp, tr, K, n_ept=n_ept, ept_mean=ept_mean)
    ref_p, ref_c, ref_s = _independent(logits, s.parent, s.cand_tokens, acc["path"],
                                       acc["accept_len"], acc["next_token"], tp, tr, K, n_ept,
                                       ept_mean)
    assert (r["status"] == 0).all()
    np.testing.assert_array_equal(r["next_state"], ref_s)
    np.testing.assert_array_equal(r["next_parent"], ref_p)
    np.testing.assert_array_equal(r["next_cand"], ref_c)


def test_templates_respect_the_state_depth_rule():
    tp, tr = W.make_tree_templates(5, 64, 4, np.random.default_rng(2))
    for k in range(5):
        depth = {0: 0}
        for i in range(1, 64):
            assert 0 <= tp[k, i] < i
            if tr[k, i] >= 0:
                assert tp[k, i] == 0 or tr[k, tp[k, i]] >= 0
                depth[i] = depth[tp[k, i]] + 1
                assert depth[i] <= k
        assert k == 0 or max(depth.values()) >= 1    # every state with k >= 1 has guesses


def test_next_tree_errors():
    parent = np.array([[-1, 0, 1], [-1, 0, 1]])
    cand = np.array([[3, -1, -1], [3, -1, -1]])
    logits = np.zeros((2, 3, 4), np.float32)
    path = np.array([[0, -1, -1], [0, -1, -1]])
    tp = np.array([[-1, 0, 1], [-1, 0, 1]])
    bad_rank = np.array([[0, -1, -1], [0, 7, -1]])      # state 1 asks for rank 7 of K = 2
    r = oracle.next_tree(logits, parent, cand, path, np.array([1, 0]), np.array([1, 1]), tp,
                         bad_rank, K=2)
    assert r["status"].tolist() == [3, 3]                # rank outside K; failed acceptance
    assert (r["next_parent"] == -1).all() and (r["next_state"] == -1).all()
    deep = np.array([[0, -1, -1], [0, 0, 0]])           # state 1 with a depth-2 candidate
    r = oracle.next_tree(logits, parent, cand, path, np.array([1, 1]), np.array([1, 1]), tp,
                         deep, K=2)
    assert r["status"].tolist() == [3, 3]
    ok = np.array([[0, -1, -1], [0, 1, -1]])
    r = oracle.next_tree(logits, parent, cand, path, np.array([1, 1]), np.array([1, 2]), tp, ok,
                         K=2)
    assert r["status"].tolist() == [0, 0] and r["next_state"].tolist() == [1, 1]
    assert r["next_cand"].tolist() == [[1, 1, -1], [2, 1, -1]]   # c_1 logits all 0: rank 1 is token 1
