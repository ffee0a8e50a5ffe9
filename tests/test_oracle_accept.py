"""Pins for the oracle's acceptance rule (Section 3: exact-matching
verification and acceptance of the longest validated path), node argmax,
bf16 rounding and KV compaction.

Expected values come from: hand-worked cases (tests/golden), an exhaustive
enumeration of root-to-node paths written top-down (a formulation distinct
from the oracle's bottom-up recursion), Proposition 1 of the appendix (the
expected number of accepted tokens of a tree), numpy.argmax, and torch's
bf16 conversion."""
import itertools
import json
import os

import numpy as np
import pytest
import torch

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------- worked examples

def test_hand_worked_examples():
    with open(os.path.join(GOLDEN, "accept_worked_examples.json")) as f:
        spec = json.load(f)
    for case in spec["cases"]:
        T = len(case["parent"])
        r = oracle.accept_path(np.array([case["argmax"]]), np.array([case["cand_tokens"]]),
                               np.array([case["parent"]]), np.array([case["prefix_len"]]),
                               case["V"], case["S_max"])
        e = case["expect"]
        path = e["path"] + [-1] * (T - len(e["path"]))
        assert r["accept_len"][0] == e["accept_len"], case["name"]
        assert r["path"][0].tolist() == path, case["name"]
        assert r["next_token"][0] == e["next_token"], case["name"]
        assert r["new_prefix_len"][0] == e["new_prefix_len"], case["name"]
        assert r["status"][0] == e["status"], case["name"]


# ----------------------------------------------------------------------------- brute force

def _all_trees(T):
    """Every topologically ordered parent array with T nodes."""
    for tail in itertools.product(*[range(i) for i in range(1, T)]):
        yield [-1] + list(tail)


def _brute_force(parent, cand, argmax, P):
    """Enumerate root-to-node paths top-down; a path is accepted when every
    step u -> c has cand[c] >= 0 and cand[c] == argmax[u]."""
    T = len(parent)
    children = [[] for _ in range(T)]
    for i in range(1, T):
        children[parent[i]].append(i)
    best = [0]
    stack = [[0]]
    while stack:
        path = stack.pop()
        u = path[-1]
        if len(path) > len(best) or (len(path) == len(best) and u < best[-1]):
            best = path
        for c in children[u]:
            if cand[c] >= 0 and cand[c] == argmax[u]:
                stack.append(path + [c])
    return len(best), best, argmax[best[-1]], P + len(best)


@pytest.mark.parametrize("T", [1, 2, 3, 4, 5, 6, 7])
def test_exhaustive_small_trees(T):
    rng = np.random.default_rng(T)
    V = 4
    parents, cands, tops = [], [], []
    for parent in _all_trees(T):
        for ok in itertools.product([0, 1], repeat=T - 1):
            top = rng.integers(0, V, size=T)
            cand = np.empty(T, np.int64)
            cand[0] = rng.integers(0, V)
            for i in range(1, T):
                if ok[i - 1]:
                    cand[i] = top[parent[i]]
                elif rng.random() < 0.5:
                    cand[i] = -1                              # prompt-token node
                else:
                    cand[i] = (top[parent[i]] + 1 + rng.integers(0, V - 1)) % V   # mismatch
            parents.append(parent)
            cands.append(cand)
            tops.append(top)
    parents, cands, tops = np.array(parents), np.array(cands), np.array(tops)
    B = len(parents)
    P = rng.integers(0, 50, size=B)
    r = oracle.accept_path(tops, cands, parents, P, V, 1000)
    assert (r["status"] == 0).all()
    for b in range(B):
        n, path, nxt, newp = _brute_force(parents[b], cands[b], tops[b], int(P[b]))
        assert r["accept_len"][b] == n
        assert r["path"][b, :n].tolist() == path
        assert (r["path"][b, n:] == -1).all()
        assert r["next_token"][b] == nxt
        assert r["new_prefix_len"][b] == newp


# ----------------------------------------------------------------------------- Proposition 1

def test_proposition_1_expected_accepted_tokens():
    """Appendix A, Proposition 1: with acceptance probability p_i at each path
    position, the expected number of accepted candidate tokens of a tree is
    sum over candidates v of prod_{i in Path(v)} p_i.  Here the model's top-1
    token at a node is its k-th ranked child's token with probability
    rank_p[k] (siblings carry distinct tokens), so the accepted candidates form
    one path and accept_len - 1 counts them."""
    rank_p = [0.45, 0.2, 0.1, 0.05]
    parent = [-1, 0, 0, 0, 1, 1, 2, 4, 4, 5, 7, 0]
    prompt = {11}                          # a prompt-token child of the root
    T = len(parent)
    children = [[c for c in range(1, T) if parent[c] == u] for u in range(T)]
    rank = {}
    for u in range(T):
        for k, c in enumerate([c for c in children[u] if c not in prompt]):
            rank[c] = k
    # closed form of Proposition 1
    f = 0.0
    for v in range(1, T):
        if v in prompt:
            continue
        prob, a = 1.0, v
        while a > 0:
            prob *= rank_p[rank[a]]
            a = parent[a]
        f += prob
    # simulation through the oracle
    N = 40000
    rng = np.random.default_rng(123)
    V = 32
    cand = np.zeros((N, T), np.int64)
    top = np.zeros((N, T), np.int64)
    for c in range(1, T):
        cand[:, c] = -1 if c in prompt else 1 + rank[c]     # distinct among siblings
    for u in range(T):
        kids = [c for c in children[u] if c not in prompt]
        probs = rank_p[:len(kids)]
        draw = rng.random(N)
        choice = np.full(N, 0)                              # token 0: matches no child
        acc = 0.0
        for k, p in enumerate(probs):
            choice = np.where((draw >= acc) & (draw < acc + p), 1 + k, choice)
            acc += p
        top[:, u] = choice
    r = oracle.accept_path(top, cand, np.tile(parent, (N, 1)), np.zeros(N), V, 100)
    got = r["accept_len"] - 1.0
    sigma = got.std() / np.sqrt(N)
    assert abs(got.mean() - f) < 4 * sigma, (got.mean(), f, sigma)


# ----------------------------------------------------------------------------- error handling

def test_rejects_bad_tokens_and_prefix():
    parent = np.array([[-1, 0, 1]] * 4)
    cand = np.array([[2, 3, -1], [9, 3, -1], [2, -2, -1], [2, 3, -1]])
    top = np.array([[3, 0, 0]] * 4)
    r = oracle.accept_path(top, cand, parent, np.array([0, 0, 0, -1]), 8, 10)
    assert r["status"].tolist() == [0, 3, 3, 4]
    assert r["accept_len"].tolist() == [2, 0, 0, 0]
    assert r["new_prefix_len"].tolist() == [2, 0, 0, -1]


# ----------------------------------------------------------------------------- argmax

def test_argmax_matches_numpy_random():
    rng = np.random.default_rng(0)
    x = rng.standard_normal((64, 1000)).astype(np.float32)
    np.testing.assert_array_equal(oracle.node_argmax(x), np.argmax(x, axis=1))


def test_argmax_ties_nan_signed_zero():
    rows = []
    a = np.zeros(37, np.float32) - 1; a[[5, 20]] = 3.0; rows.append(a)          # tie -> 5
    a = np.zeros(37, np.float32) - 1; a[9] = np.nan; a[3] = np.nan; a[1] = 9; rows.append(a)
    a = np.full(37, -2.0, np.float32); a[4] = -0.0; a[2] = 0.0; rows.append(a)    # +-0 tie -> 2
    a = np.full(37, -2.0, np.float32); a[4] = 0.0; a[2] = -0.0; rows.append(a)
    a = np.full(37, 1.5, np.float32); rows.append(a)                            # all equal -> 0
    a = np.zeros(37, np.float32); a[30] = np.inf; a[31] = np.inf; rows.append(a)
    a = np.zeros(37, np.float32); a[0] = np.nan; rows.append(a)
    a = np.full(37, -np.inf, np.float32); a[36] = -1e30; rows.append(a)
    x = np.stack(rows)
    np.testing.assert_array_equal(oracle.node_argmax(x), np.argmax(x, axis=1))
    np.testing.assert_array_equal(oracle.node_argmax(x[:, :1]), np.zeros(len(rows)))


# ----------------------------------------------------------------------------- bf16 rounding

def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(1)
    x = np.concatenate([
        rng.standard_normal(10000).astype(np.float32) * np.float32(10.0) ** rng.integers(-40, 38, 10000).astype(np.float32),
        np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 1 + 2 ** -8 + 2 ** -20,
                  3.3895314e38, 3.4028235e38, -3.4028235e38, 1e-45, 1.17e-38, 0.0, -0.0,
                  np.inf, -np.inf], np.float32)])
    x = x[np.isfinite(x) | np.isinf(x)]
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.round_bf16(x)
    np.testing.assert_array_equal(got, want)
    nan = oracle.round_bf16(np.array([np.nan, -np.nan], np.float32))
    assert ((nan & 0x7f80) == 0x7f80).all() and ((nan & 0x7f) != 0).all()


# ----------------------------------------------------------------------------- compaction

def test_kv_compact_copies_rows_and_nothing_else():
    rng = np.random.default_rng(5)
    L, B, H, T, D, S = 2, 3, 2, 6, 8, 20
    kc = rng.integers(0, 65535, (L, B, H, S, D)).astype(np.uint16)
    vc = rng.integers(0, 65535, (L, B, H, S, D)).astype(np.uint16)
    kt = rng.integers(0, 65535, (L, B, H, T, D)).astype(np.uint16)
    vt = rng.integers(0, 65535, (L, B, H, T, D)).astype(np.uint16)
    path = np.array([[0, 2, 5, -1, -1, -1], [0, -1, -1, -1, -1, -1], [-1] * 6], np.int32)
    acc = np.array([3, 1, 0], np.int32)
    pre = np.array([4, 19, 7], np.int32)
    k2, v2 = oracle.kv_compact(kc, vc, kt, vt, path, acc, pre)
    ek, ev = kc.copy(), vc.copy()
    for b in range(B):
        for j in range(acc[b]):
            ek[:, b, :, pre[b] + j] = kt[:, b, :, path[b, j]]
            ev[:, b, :, pre[b] + j] = vt[:, b, :, path[b, j]]
    np.testing.assert_array_equal(k2, ek)
    np.testing.assert_array_equal(v2, ev)
    # fp32 storage is copied bit for bit too
    k3, _ = oracle.kv_compact(kc.view(np.float32), vc.view(np.float32), kt.view(np.float32),
                              vt.view(np.float32), path, acc, pre // 1)
    assert k3.dtype == np.float32
