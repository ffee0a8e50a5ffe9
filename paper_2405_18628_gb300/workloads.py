"""Seeded synthetic workloads for the PPD verification step.

This module only *draws inputs*: token trees, candidate token ids, Q/K/V
tensors and node logits.  It contains none of the verification arithmetic
(no attention, no argmax, no acceptance rule); the CUDA path and the CPU
oracle both consume what it produces.

Shapes follow the paper's evaluation models (MobileLLaMA-1.4B, Vicuna-7B,
Vicuna-13B; Section 5 "Models and testbeds") and its customised sparse tree:
a tree of candidate ("guess") tokens where each candidate carries a chain of
prompt tokens below it (Section 4.1).  Tree sizes sit between the paper's
tree-input lengths of 40..285 tokens (Table 1, column S_input).

Logits are drawn i.i.d. N(0,1) per row with the position of the row maximum
drawn first (order-statistics sampling), so the generator knows every row's
top token without ever scanning a row.  Candidate token ids copy the parent's
top token with the configured match rate, else are uniform over the vocab.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Tuple

import numpy as np

SEED_BASE = 2405_18628


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic verification-step workload (sizes per the paper's models)."""

    name: str
    L: int            # layers
    B: int            # batch (sequences)
    H: int            # heads (MHA: K/V heads == query heads)
    D: int            # head dim
    P: int            # KV prefix length (cached tokens) per sequence
    T: int            # tree tokens per sequence (root + candidates + prompt tokens)
    V: int            # vocab size
    n_cand: int       # candidate nodes including the root
    max_depth: int    # depth cap of candidate nodes (root depth 0)
    chains: str       # prompt-chain recipe, see _chain_lengths
    match_rate: float
    dtype: str = "bf16"   # storage type of Q/K/V: "bf16" or "f32"
    seed: int = SEED_BASE

    @property
    def S_max(self) -> int:
        """Cache capacity: the prefix plus room for every tree token."""
        return self.P + self.T


WORKLOADS = {
    "tiny": Workload("tiny", L=1, B=1, H=4, D=64, P=128, T=48, V=1024, n_cand=16,
                     max_depth=4, chains="every2", match_rate=0.5, seed=SEED_BASE + 0),
    "tiny_f32": Workload("tiny_f32", L=1, B=1, H=4, D=64, P=128, T=48, V=1024, n_cand=16,
                         max_depth=4, chains="every2", match_rate=0.5, dtype="f32",
                         seed=SEED_BASE + 0),
    "mobilellama": Workload("mobilellama", L=24, B=1, H=16, D=128, P=512, T=64, V=32000,
                            n_cand=24, max_depth=5, chains="fill3", match_rate=0.6,
                            seed=SEED_BASE + 1),
    "vicuna7b": Workload("vicuna7b", L=32, B=1, H=32, D=128, P=2048, T=64, V=32000,
                         n_cand=40, max_depth=6, chains="leaf1to3", match_rate=0.6,
                         seed=SEED_BASE + 2),
    "vicuna13b": Workload("vicuna13b", L=40, B=1, H=40, D=128, P=4096, T=96, V=32000,
                          n_cand=60, max_depth=6, chains="fill3", match_rate=0.5,
                          seed=SEED_BASE + 3),
}
for _t in (16, 32, 64, 128):
    WORKLOADS[f"sweep_t{_t}"] = Workload(
        f"sweep_t{_t}", L=32, B=8, H=32, D=128, P=16384, T=_t, V=32000, n_cand=_t // 4,
        max_depth=8, chains="every3", match_rate=0.6, seed=SEED_BASE + 4)


def scaled(w: Workload, **kw) -> Workload:
    """A copy of `w` with some sizes replaced (used for small parity cases)."""
    return dataclasses.replace(w, **kw)


# ----------------------------------------------------------------------------- trees

def _candidate_tree(rng: np.random.Generator, n_cand: int, max_depth: int):
    """Random candidate tree: parent of node i uniform over earlier nodes whose
    depth is below the cap (so every candidate has depth <= max_depth)."""
    parent = [-1]
    depth = [0]
    for i in range(1, n_cand):
        eligible = [j for j in range(i) if depth[j] < max_depth]
        p = eligible[int(rng.integers(len(eligible)))]
        parent.append(p)
        depth.append(depth[p] + 1)
    return parent, depth


def _chain_lengths(rng, recipe: str, parent, depth, n_prompt: int) -> List[Tuple[int, int]]:
    """Decide (anchor candidate, chain length) pairs totalling exactly n_prompt."""
    n_cand = len(parent)
    has_child = [False] * n_cand
    for p in parent[1:]:
        has_child[p] = True
    leaves = [i for i in range(n_cand) if not has_child[i]]
    internal_deep_first = sorted((i for i in range(n_cand) if has_child[i]),
                                 key=lambda i: (-depth[i], i))
    if recipe.startswith("every"):
        c = int(recipe[len("every"):])
        return [(i, c) for i in range(n_cand)]
    if recipe.startswith("ept"):
        # "ept<n>x<c>": n ensemble chains of c prompt tokens on every candidate
        n, c = (int(x) for x in recipe[len("ept"):].split("x"))
        return [(i, c) for i in range(n_cand) for _ in range(n)]
    if recipe == "fill3":
        # chains of 3 on leaves in index order, then on the deepest internal
        # nodes; the last chain is truncated to hit the total exactly
        out, left = [], n_prompt
        for a in leaves + internal_deep_first:
            if left <= 0:
                break
            c = min(3, left)
            out.append((a, c))
            left -= c
        return out
    if recipe == "leaf1to3":
        # 1..3 prompt tokens per leaf (drawn), clipped to the total; any
        # remainder is handed out round-robin (up to 3 per anchor), first to
        # leaves, then to the deepest internal nodes
        want = {a: 1 + int(rng.integers(3)) for a in leaves}
        out, left = {}, n_prompt
        for a in leaves:
            c = min(want[a], left)
            if c > 0:
                out[a] = c
                left -= c
        for pool in (leaves, internal_deep_first):
            progress = True
            while left > 0 and progress:
                progress = False
                for a in pool:
                    if left > 0 and out.get(a, 0) < 3:
                        out[a] = out.get(a, 0) + 1
                        left -= 1
                        progress = True
        return sorted(out.items())
    raise ValueError(f"unknown chain recipe {recipe!r}")


def make_tree_templates(n_states: int, T_next: int, K: int, rng: np.random.Generator,
                        n_ept: int = 1):
    """Next-step tree templates, one per state k = 0..n_states-1 (the paper's
    T_k, Appendix: the candidate subtree of T_k is at most k deep).  Node 0 is
    the root; candidate nodes carry the rank (0..K-1) of the guess they take at
    their depth, prompt nodes rank -1.  Candidates: up to K children of the root
    at depth 1, then at each further depth up to K children of the depth's
    rank-0 node and of one other random candidate, within a budget of
    T_next // 4 candidates; n_ept prompt chains of up to n_states-1 tokens each
    then hang below the root and the candidates, in index order, filling
    exactly T_next nodes.  Returns (parent, rank), both int32 [n_states,
    T_next]."""
    m = n_states - 1
    parent = np.full((n_states, T_next), -1, np.int32)
    rank = np.full((n_states, T_next), -1, np.int32)
    for k in range(n_states):
        par, rk, depth = [-1], [0], [0]
        budget = max(1, T_next // 4)
        level = [0]
        for d in range(1, k + 1):
            anchors = [level[0]]
            if len(level) > 1:
                anchors.append(level[1 + int(rng.integers(len(level) - 1))])
            nxt = []
            for a in anchors:
                for r in range(K):
                    if len(par) >= budget:
                        break
                    par.append(a)
                    rk.append(r)
                    depth.append(d)
                    nxt.append(len(par) - 1)
            if not nxt:
                break
            level = nxt
        n_cand = len(par)
        for a in range(n_cand):
            for _ in range(n_ept):
                prev = a
                for _ in range(m):
                    if len(par) >= T_next:
                        break
                    par.append(prev)
                    rk.append(-1)
                    prev = len(par) - 1
        while len(par) < T_next:                  # more room than chains: extend the root's
            par.append(len(par) - 1 if rk[-1] == -1 else 0)
            rk.append(-1)
        parent[k] = par[:T_next]
        rank[k] = rk[:T_next]
    return parent, rank


def make_tree(rng: np.random.Generator, w: Workload):
    """One sequence's tree.  Returns (parent int32[T], is_prompt bool[T]).

    Nodes 0..n_cand-1 are the root and candidates (topological order), then the
    prompt-token chains: the first prompt node of a chain hangs under its
    anchor candidate and every further one under the previous prompt node.
    """
    parent, depth = _candidate_tree(rng, w.n_cand, w.max_depth)
    chains = _chain_lengths(rng, w.chains, parent, depth, w.T - w.n_cand)
    is_prompt = [False] * w.n_cand
    for anchor, length in chains:
        prev = anchor
        for _ in range(length):
            parent.append(prev)
            is_prompt.append(True)
            prev = len(parent) - 1
    if len(parent) != w.T:
        raise AssertionError(f"{w.name}: tree has {len(parent)} nodes, want {w.T}")
    return np.asarray(parent, np.int32), np.asarray(is_prompt, bool)


# ----------------------------------------------------------------------------- logits

def planted_logits(rng: np.random.Generator, rows: int, V: int):
    """Rows of i.i.d. N(0,1) fp32 logits together with each row's top index.

    The row maximum is drawn first from its distribution (CDF Phi(x)^V) and put
    at a uniformly drawn position; the other V-1 entries are N(0,1) draws
    conditioned to lie below it.  The joint law equals V i.i.d. N(0,1) draws,
    and the top index is known by construction (ties are excluded in fp32).
    """
    from scipy.special import ndtr, ndtri

    top = rng.integers(0, V, size=rows).astype(np.int64)
    mx = ndtri(rng.random(rows) ** (1.0 / V))
    mx32 = mx.astype(np.float32)
    below = np.nextafter(mx32, np.float32(-np.inf))
    out = np.empty((rows, V), np.float32)
    chunk = max(1, (1 << 22) // max(V, 1))
    cols = np.arange(V)
    for r0 in range(0, rows, chunk):
        r1 = min(rows, r0 + chunk)
        u = rng.random((r1 - r0, V - 1))
        rest = ndtri(u * ndtr(mx[r0:r1, None])).astype(np.float32)
        rest = np.minimum(rest, below[r0:r1, None])
        full = np.concatenate([rest, mx32[r0:r1, None]], axis=1)
        t = top[r0:r1, None]
        src = np.where(cols[None, :] < t, cols[None, :],
                       np.where(cols[None, :] == t, V - 1, cols[None, :] - 1))
        out[r0:r1] = np.take_along_axis(full, src, axis=1)
    return out, top.astype(np.int32)


# ----------------------------------------------------------------------------- step inputs

@dataclasses.dataclass
class StepInputs:
    """Host-side integer/logit inputs of one verification step."""

    parent: np.ndarray        # int32 [B, T]
    cand_tokens: np.ndarray   # int32 [B, T]  (-1 marks prompt-token nodes)
    prefix_len: np.ndarray    # int32 [B]
    logits: np.ndarray        # float32 [B, T, V]
    top: np.ndarray           # int32 [B, T]  planted top token of each logits row


def make_step_inputs(w: Workload, seed: Optional[int] = None,
                     prefix_len: Optional[np.ndarray] = None) -> StepInputs:
    """Trees, candidate ids, prefix lengths and logits for every sequence."""
    rng = np.random.Generator(np.random.PCG64(w.seed if seed is None else seed))
    parents, prompts = [], []
    for _ in range(w.B):
        p, isp = make_tree(rng, w)
        parents.append(p)
        prompts.append(isp)
    parent = np.stack(parents)
    is_prompt = np.stack(prompts)
    logits, top = planted_logits(rng, w.B * w.T, w.V)
    logits = logits.reshape(w.B, w.T, w.V)
    top = top.reshape(w.B, w.T)
    cand = np.empty((w.B, w.T), np.int32)
    for b in range(w.B):
        cand[b, 0] = int(rng.integers(w.V))          # root: the last accepted token
        for i in range(1, w.T):
            if is_prompt[b, i]:
                cand[b, i] = -1
            elif rng.random() < w.match_rate:
                cand[b, i] = top[b, parent[b, i]]
            else:
                cand[b, i] = int(rng.integers(w.V))
    if prefix_len is None:
        prefix_len = np.full(w.B, w.P, np.int32)
    return StepInputs(parent=parent, cand_tokens=cand,
                      prefix_len=np.asarray(prefix_len, np.int32), logits=logits, top=top)


def make_tensors(w: Workload, device="cpu", seed: Optional[int] = None,
                 poison_tail: bool = False, S_max: Optional[int] = None):
    """Q, K/V cache and tree K/V, N(0,1) then stored as bf16 (or fp32).

    Drawn with a seeded torch generator on `device`.  With `poison_tail`, cache
    rows at or beyond each sequence's prefix length hold NaN so that any use
    of an invisible row shows up in the output.
    """
    import torch

    S = w.S_max if S_max is None else S_max
    g = torch.Generator(device=device)
    g.manual_seed((w.seed if seed is None else seed) * 7 + 1)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32

    def draw(*shape):
        # drawn one layer at a time so the fp32 temporary stays small
        out = torch.empty(shape, dtype=dt, device=device)
        for l in range(shape[0]):
            x = torch.empty(shape[1:], dtype=torch.float32, device=device)
            x.normal_(generator=g)
            out[l].copy_(x)
        return out

    q = draw(w.L, w.B, w.H, w.T, w.D)
    k_cache = draw(w.L, w.B, w.H, S, w.D)
    v_cache = draw(w.L, w.B, w.H, S, w.D)
    k_tree = draw(w.L, w.B, w.H, w.T, w.D)
    v_tree = draw(w.L, w.B, w.H, w.T, w.D)
    if poison_tail:
        k_cache[:, :, :, w.P:, :] = float("nan")
        v_cache[:, :, :, w.P:, :] = float("nan")
    return dict(q=q, k_cache=k_cache, v_cache=v_cache, k_tree=k_tree, v_tree=v_tree)


def poison_cache_tail(k_cache, v_cache, prefix_len):
    """Set cache rows [prefix_len[b], S_max) of every sequence to NaN."""
    for b, p in enumerate(np.asarray(prefix_len).tolist()):
        k_cache[:, b, :, p:, :] = float("nan")
        v_cache[:, b, :, p:, :] = float("nan")
