"""Pins for the oracle's typical acceptance (Section 3 step (2) names typical
acceptance as the second verification scheme; the rule tested is
p(tok) > min(epsilon, delta * exp(-H)) under softmax(logits / temperature)).

Expected values come from scipy's logsumexp / softmax / entropy (library
routines, not the oracle's loops), closed forms for uniform and two-level
logits, the exact-matching oracle in the zero-temperature limit, degenerate
thresholds (zero: every candidate passes; one: none does), invariance under a
common scaling of logits and temperature, and an exhaustive top-down
enumeration of root-to-node paths on small trees."""
import itertools

import numpy as np
import pytest
from scipy.special import logsumexp, softmax
from scipy.stats import entropy

import oracle


def _tree(rng, T):
    return np.array([-1] + [int(rng.integers(0, i)) for i in range(1, T)])


# ----------------------------------------------------------------------------- statistics

@pytest.mark.parametrize("tau", [0.25, 1.0, 3.0])
def test_node_stats_match_scipy(tau):
    rng = np.random.default_rng(11)
    x = (rng.standard_normal((5, 777)) * 2.0).astype(np.float32)
    lse, ent = oracle.node_stats(x, tau)
    y = x.astype(np.float64) / tau
    np.testing.assert_allclose(lse, logsumexp(y, axis=-1), rtol=1e-13)
    np.testing.assert_allclose(ent, entropy(softmax(y, axis=-1), axis=-1), rtol=1e-11)


def test_node_stats_closed_forms():
    V = 1000
    # uniform: lse = c / tau + log V, H = log V
    x = np.full((1, V), 2.5, np.float32)
    lse, ent = oracle.node_stats(x, 0.5)
    assert lse[0] == pytest.approx(5.0 + np.log(V), rel=1e-14)
    assert ent[0] == pytest.approx(np.log(V), rel=1e-12)
    # one logit a above V-1 zeros: Z = e^a + V - 1, H = log Z - a e^a / Z
    a = 3.0
    x = np.zeros((1, V), np.float32)
    x[0, 17] = a
    lse, ent = oracle.node_stats(x, 1.0)
    Z = np.exp(a) + V - 1
    assert lse[0] == pytest.approx(np.log(Z), rel=1e-14)
    assert ent[0] == pytest.approx(np.log(Z) - a * np.exp(a) / Z, rel=1e-12)


def test_node_stats_nan_and_neg_inf():
    x = np.zeros((3, 8), np.float32)
    x[0, 3] = np.nan
    x[1, :4] = -np.inf                      # impossible tokens: probability 0
    lse, ent = oracle.node_stats(x, 1.0)
    assert np.isnan(lse[0]) and np.isnan(ent[0])
    assert lse[1] == pytest.approx(np.log(4.0)) and ent[1] == pytest.approx(np.log(4.0))
    assert lse[2] == pytest.approx(np.log(8.0)) and ent[2] == pytest.approx(np.log(8.0))


# ----------------------------------------------------------------------------- acceptance

def _random_case(rng, B, T, V, match=0.5, prompt=0.2):
    logits = (rng.standard_normal((B, T, V)) * 1.5).astype(np.float32)
    parent = np.stack([_tree(rng, T) for _ in range(B)])
    top = oracle.node_argmax(logits)
    cand = rng.integers(0, V, size=(B, T))
    for b in range(B):
        for i in range(1, T):
            u = rng.random()
            if u < prompt:
                cand[b, i] = -1
            elif u < prompt + match:
                cand[b, i] = top[b, parent[b, i]]
    return logits, parent, top, cand


def test_zero_temperature_limit_is_exact_matching():
    """As the temperature goes to zero p concentrates on the argmax token, so
    with epsilon = 0.5 a candidate passes exactly when it equals its parent's
    argmax: typical acceptance reduces to exact matching."""
    rng = np.random.default_rng(3)
    B, T, V = 64, 12, 50
    logits, parent, _, cand = _random_case(rng, B, T, V, match=0.0)
    # every row's maximum 0.5 above the rest: at temperature 1e-3 p(top) = 1 - O(e^-500)
    am = logits.argmax(axis=-1)
    np.put_along_axis(logits, am[..., None],
                      np.take_along_axis(logits, am[..., None], -1) + 0.5, axis=-1)
    top = oracle.node_argmax(logits)
    for b in range(B):
        for i in range(1, T):
            if cand[b, i] >= 0 and rng.random() < 0.6:
                cand[b, i] = top[b, parent[b, i]]
    P = rng.integers(0, 40, size=B)
    ex = oracle.accept_path(top, cand, parent, P, V, 100)
    ty = oracle.typical_accept(logits, top, cand, parent, P, 100, temperature=1e-3,
                               epsilon=0.5, delta=0.5)
    for k in ("accept_len", "path", "next_token", "new_prefix_len", "status"):
        np.testing.assert_array_equal(ty[k], ex[k], err_msg=k)


def test_degenerate_thresholds():
    rng = np.random.default_rng(5)
    B, T, V = 16, 10, 40
    logits, parent, top, cand = _random_case(rng, B, T, V)
    P = np.zeros(B, np.int64)
    # threshold 0: every candidate passes; accepted = nodes whose path has no prompt node
    r = oracle.typical_accept(logits, top, cand, parent, P, 100, 1.0, 0.0, 0.5)
    for b in range(B):
        cand_only = [i for i in range(T)
                     if all(cand[b, a] >= 0 for a in _root_path(parent[b], i))]
        depth = {i: len(_root_path(parent[b], i)) for i in cand_only}
        best = min(cand_only, key=lambda i: (-depth[i], i))
        assert r["accept_len"][b] == depth[best]
        assert r["path"][b, :depth[best]].tolist() == _root_path(parent[b], best)
    # threshold 1 (epsilon 1, delta huge): p < 1 everywhere, only the root
    r = oracle.typical_accept(logits, top, cand, parent, P, 100, 1.0, 1.0, 1e30)
    assert (r["accept_len"] == 1).all()
    assert (r["next_token"] == top[:, 0]).all()


def _root_path(parent, i):
    path = []
    while i >= 0:
        path.append(int(i))
        i = parent[i]
    return path[::-1]


def test_invariant_under_common_scaling():
    """softmax(x / tau) depends on x / tau only."""
    rng = np.random.default_rng(8)
    B, T, V = 24, 9, 64
    logits, parent, top, cand = _random_case(rng, B, T, V)
    P = np.zeros(B, np.int64)
    a = oracle.typical_accept(logits, top, cand, parent, P, 50, 0.7, 0.09, 0.3)
    b = oracle.typical_accept(logits * 4.0, top, cand, parent, P, 50, 2.8, 0.09, 0.3)
    for k in ("accept_len", "path", "next_token"):
        np.testing.assert_array_equal(a[k], b[k])
    np.testing.assert_allclose(a["p_tok"], b["p_tok"], rtol=1e-12, equal_nan=True)


@pytest.mark.parametrize("T", [2, 3, 4, 5])
def test_exhaustive_small_trees_typical(T):
    """Every topologically ordered tree of T nodes, random logits: top-down
    path enumeration with the test p_t > min(eps, delta e^-H) evaluated by
    scipy."""
    rng = np.random.default_rng(20 + T)
    V, tau, eps, delta = 6, 0.8, 0.2, 0.5
    trees = [[-1] + list(t) for t in itertools.product(*[range(i) for i in range(1, T)])]
    for parent in trees:
        for _ in range(6):
            logits = (rng.standard_normal((1, T, V)) * 1.2).astype(np.float32)
            cand = rng.integers(-1, V, size=(1, T))
            cand[0, 0] = rng.integers(0, V)
            top = oracle.node_argmax(logits)
            r = oracle.typical_accept(logits, top, cand, np.array([parent]), np.array([3]), 50,
                                      tau, eps, delta)
            p = softmax(logits[0].astype(np.float64) / tau, axis=-1)
            H = entropy(p, axis=-1)

            def passes(u, c):
                return cand[0, c] >= 0 and p[u, cand[0, c]] > min(eps, delta * np.exp(-H[u]))

            children = [[c for c in range(1, T) if parent[c] == u] for u in range(T)]
            best, stack = [0], [[0]]
            while stack:
                path = stack.pop()
                u = path[-1]
                if len(path) > len(best) or (len(path) == len(best) and u < best[-1]):
                    best = path
                stack += [path + [c] for c in children[u] if passes(u, c)]
            assert r["accept_len"][0] == len(best)
            assert r["path"][0, :len(best)].tolist() == best
            assert r["next_token"][0] == top[0, best[-1]]
            assert r["new_prefix_len"][0] == 3 + len(best)


def test_typical_rejects_bad_arguments_and_sequences():
    logits = np.zeros((2, 3, 4), np.float32)
    parent = np.array([[-1, 0, 1], [-1, 2, 0]])
    cand = np.array([[1, 2, 3], [1, 2, 3]])
    top = np.zeros((2, 3), np.int32)
    with pytest.raises(ValueError):
        oracle.typical_accept(logits, top, cand, parent, [0, 0], 10, 0.0, 0.1, 0.1)
    r = oracle.typical_accept(logits, top, cand, parent, [0, 0], 10, 1.0, 0.1, 0.1)
    assert r["status"].tolist() == [0, 3]
    assert np.isnan(r["p_tok"][1]).all() and np.isnan(r["p_tok"][0, 0])
    # uniform over 4 tokens: p = 1/4, H = log 4, threshold min(0.1, 0.1/4) = 0.025
    np.testing.assert_allclose(r["p_tok"][0, 1:], 0.25)
    np.testing.assert_allclose(r["threshold"][0, 1:], 0.025)
    assert r["accept_len"].tolist() == [3, 0]
