"""Pins for the oracle's tree-masked attention (Section 3 step (1), Section
4.1: each tree token attends to the cached prefix, its tree ancestors and
itself).  Every expected value here comes from a library routine
(torch scaled_dot_product_attention in fp64 on the CPU, torch.logsumexp), a
closed form, an invariant, or a brute-force ancestor relation, never from
the oracle itself."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import workloads as W


def _bf16(shape, gen):
    return torch.randn(shape, generator=gen, dtype=torch.float32).to(torch.bfloat16)


def _case(L=1, B=1, H=2, T=8, D=64, P=16, S_max=None, seed=0):
    g = torch.Generator().manual_seed(seed)
    S_max = P + T if S_max is None else S_max
    return dict(q=_bf16((L, B, H, T, D), g), k_cache=_bf16((L, B, H, S_max, D), g),
                v_cache=_bf16((L, B, H, S_max, D), g), k_tree=_bf16((L, B, H, T, D), g),
                v_tree=_bf16((L, B, H, T, D), g))


def _ancestor_mask(parent):
    """Brute-force visibility: reflexive-transitive closure of the child->parent
    relation by repeated boolean matrix products (independent of any walk)."""
    T = len(parent)
    A = np.eye(T, dtype=bool)
    for i in range(1, T):
        A[i, parent[i]] = True
    R = A.copy()
    for _ in range(T):
        R = (R.astype(np.int64) @ A.astype(np.int64)) > 0
    return R      # R[i, j]: j is i or an ancestor of i


def _sdpa_reference(t, prefix_len, parent, scale=None):
    """fp64 SDPA over [prefix ; tree] keys with an explicit boolean mask."""
    q = t["q"].double()
    L, B, H, T, D = q.shape
    outs, lses = [], []
    for b in range(B):
        P = int(prefix_len[b])
        k = torch.cat([t["k_cache"][:, b, :, :P].double(), t["k_tree"][:, b].double()], dim=2)
        v = torch.cat([t["v_cache"][:, b, :, :P].double(), t["v_tree"][:, b].double()], dim=2)
        anc = torch.from_numpy(_ancestor_mask(parent[b]))
        mask = torch.cat([torch.ones(T, P, dtype=torch.bool), anc], dim=1)
        o = torch.nn.functional.scaled_dot_product_attention(q[:, b], k, v, attn_mask=mask,
                                                             scale=scale)
        s = (q[:, b] @ k.transpose(-1, -2)) * (scale if scale else D ** -0.5)
        s = s.masked_fill(~mask, float("-inf"))
        outs.append(o)
        lses.append(torch.logsumexp(s, dim=-1))
    # back to [L,B,H,T,D] flattened over (l,b,h) units
    o = torch.stack(outs, dim=1).reshape(L * B * H, T, D)
    lse = torch.stack(lses, dim=1).reshape(L * B * H, T)
    return o.numpy(), lse.numpy()


def _run(t, prefix_len, parent, **kw):
    return oracle.tree_attention(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                 np.asarray(prefix_len, np.int32), np.asarray(parent, np.int32),
                                 **kw)


def test_chain_tree_is_causal_attention():
    """parent[i] = i-1 and no prefix: exactly causal self-attention."""
    T = 12
    t = _case(T=T, P=0, H=3)
    parent = np.array([[-1] + list(range(T - 1))], np.int32)
    out, lse, rs, st = _run(t, [0], parent)
    ref = torch.nn.functional.scaled_dot_product_attention(
        t["q"][:, 0].double(), t["k_tree"][:, 0].double(), t["v_tree"][:, 0].double(),
        is_causal=True).reshape(-1, T, 64).numpy()
    assert (st == 0).all()
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_chain_with_prefix_matches_masked_sdpa():
    T, P = 9, 21
    t = _case(T=T, P=P, H=2, L=2)
    parent = np.array([[-1] + list(range(T - 1))], np.int32)
    out, lse, _, _ = _run(t, [P], parent)
    ref, ref_lse = _sdpa_reference(t, [P], parent)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=0, atol=1e-12)


@pytest.mark.parametrize("seed", range(4))
def test_random_tree_matches_masked_sdpa(seed):
    w = W.scaled(W.WORKLOADS["tiny"], B=3, H=2, L=2, P=37)
    s = W.make_step_inputs(w, seed=seed, prefix_len=np.array([37, 0, 5], np.int32))
    t = _case(L=2, B=3, H=2, T=w.T, D=64, P=37, seed=seed)
    out, lse, rs, st = _run(t, s.prefix_len, s.parent)
    ref, ref_lse = _sdpa_reference(t, s.prefix_len, s.parent)
    assert (st == 0).all()
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=0, atol=1e-12)
    np.testing.assert_allclose(rs, 1.0, rtol=0, atol=1e-12)


def test_explicit_scale():
    T = 6
    t = _case(T=T, P=4)
    parent = np.array([[-1, 0, 0, 1, 2, 2]], np.int32)
    out, _, _, _ = _run(t, [4], parent, scale=0.3)
    ref, _ = _sdpa_reference(t, [4], parent, scale=0.3)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-12)


def test_single_token_is_decode_attention():
    """T = 1: plain decode attention of one query over prefix + itself."""
    t = _case(T=1, P=50, H=4)
    out, _, _, _ = _run(t, [50], np.array([[-1]], np.int32))
    q = t["q"][:, 0].double()
    k = torch.cat([t["k_cache"][:, 0, :, :50], t["k_tree"][:, 0]], 2).double()
    v = torch.cat([t["v_cache"][:, 0, :, :50], t["v_tree"][:, 0]], 2).double()
    ref = torch.softmax(q @ k.transpose(-1, -2) / 8.0, -1) @ v
    np.testing.assert_allclose(out, ref.reshape(4, 1, 64).numpy(), rtol=0, atol=1e-12)


def test_sibling_permutation_invariance():
    """Relabelling nodes (keeping parent < child) permutes the outputs only."""
    parent = np.array([-1, 0, 0, 1, 1, 2, 3, 5], np.int32)
    t = _case(T=8, P=10, H=2)
    out, _, _, _ = _run(t, [10], parent[None])
    # swap the subtrees of siblings 1 and 2: new order 0,2,1,5,3,4,7,6
    perm = np.array([0, 2, 1, 5, 3, 4, 7, 6])        # new index k holds old node perm[k]
    inv = np.argsort(perm)
    new_parent = np.array([-1 if parent[o] < 0 else inv[parent[o]] for o in perm], np.int32)
    assert all(0 <= new_parent[i] < i for i in range(1, 8))
    t2 = dict(t)
    for k in ("q", "k_tree", "v_tree"):
        t2[k] = t[k][:, :, :, torch.from_numpy(perm)]
    out2, _, _, _ = _run(t2, [10], new_parent[None])
    np.testing.assert_allclose(out2, out[:, perm], rtol=0, atol=1e-12)


def test_identical_keys_give_mean_of_visible_values():
    T, P = 7, 11
    parent = np.array([-1, 0, 1, 0, 3, 4, 1], np.int32)
    t = _case(T=T, P=P, H=1)
    row = t["k_cache"][0, 0, 0, 0].clone()
    t["k_cache"][:] = row
    t["k_tree"][:] = row
    out, _, _, _ = _run(t, [P], parent[None])
    anc = _ancestor_mask(parent)
    for i in range(T):
        vis = torch.cat([t["v_cache"][0, 0, 0, :P], t["v_tree"][0, 0, 0][torch.from_numpy(anc[i])]])
        np.testing.assert_allclose(out[0, i], vis.double().mean(0).numpy(), rtol=0, atol=1e-12)


def test_constant_values_give_constant_output():
    t = _case(T=5, P=9, H=2)
    t["v_cache"][:] = 0.75
    t["v_tree"][:] = 0.75
    out, _, _, _ = _run(t, [9], np.array([[-1, 0, 0, 2, 2]], np.int32))
    np.testing.assert_allclose(out, 0.75, rtol=0, atol=1e-14)


def test_star_tree_sees_root_and_self():
    T, P = 6, 3
    t = _case(T=T, P=P, H=1)
    parent = np.array([[-1, 0, 0, 0, 0, 0]], np.int32)
    out, _, _, _ = _run(t, [P], parent)
    for i in range(1, T):
        keys = [0, i]
        q = t["q"][0, 0, 0, i].double()
        k = torch.cat([t["k_cache"][0, 0, 0, :P], t["k_tree"][0, 0, 0, keys]]).double()
        v = torch.cat([t["v_cache"][0, 0, 0, :P], t["v_tree"][0, 0, 0, keys]]).double()
        ref = torch.softmax(k @ q / 8.0, 0) @ v
        np.testing.assert_allclose(out[0, i], ref.numpy(), rtol=0, atol=1e-12)


def test_mask_locality_and_tail_rows_unused():
    """Changing a non-ancestor's K/V, or cache rows at/after the prefix, leaves
    an output row unchanged; changing an ancestor's K/V changes it."""
    T, P = 8, 12
    parent = np.array([-1, 0, 0, 1, 2, 3, 3, 4], np.int32)
    t = _case(T=T, P=P, H=1, S_max=P + T + 5)
    out, _, _, _ = _run(t, [P], parent[None])
    t2 = {k: v.clone() for k, v in t.items()}
    t2["k_tree"][0, 0, 0, 2] += 1.0      # node 2 is not an ancestor of 5 (path 5,3,1,0)
    t2["v_tree"][0, 0, 0, 2] -= 1.0
    t2["k_cache"][0, 0, 0, P:] = float("nan")
    t2["v_cache"][0, 0, 0, P:] = float("nan")
    out2, _, _, _ = _run(t2, [P], parent[None])
    for i in (1, 3, 5, 6):
        np.testing.assert_array_equal(out2[0, i], out[0, i])
    assert np.abs(out2[0, 2] - out[0, 2]).max() > 1e-3
    assert np.abs(out2[0, 4] - out[0, 4]).max() > 1e-3     # 4's parent is 2


def test_f32_inputs_are_rounded_to_bf16():
    t = _case(T=6, P=7, H=2)
    g = torch.Generator().manual_seed(3)
    f32 = {k: v.float() + 1e-3 * torch.randn(v.shape, generator=g) for k, v in t.items()}
    rounded = {k: v.to(torch.bfloat16) for k, v in f32.items()}   # library RNE rounding
    parent = np.array([[-1, 0, 1, 1, 0, 4]], np.int32)
    o1, _, _, _ = _run(f32, [7], parent)
    o2, _, _, _ = _run(rounded, [7], parent)
    np.testing.assert_array_equal(o1, o2)


def test_unit_subset_matches_full():
    w = W.scaled(W.WORKLOADS["tiny"], L=2, B=2, H=3, P=20)
    s = W.make_step_inputs(w)
    t = _case(L=2, B=2, H=3, T=w.T, P=20)
    full, lse, _, _ = _run(t, s.prefix_len, s.parent)
    units = [11, 0, 7]
    sub, sub_lse, _, _ = _run(t, s.prefix_len, s.parent, units=units)
    np.testing.assert_array_equal(sub, full[units])
    np.testing.assert_array_equal(sub_lse, lse[units])


def test_malformed_tree_and_prefix_flagged():
    t = _case(B=3, T=4, P=5)
    parent = np.array([[-1, 0, 1, 1], [-1, 0, 3, 1], [-1, 0, 0, 0]], np.int32)
    out, _, _, st = _run(t, [5, 5, 99], parent)
    assert st.tolist() == [0, 3, 4]
    H = 2
    assert np.isfinite(out[0:H]).all()
    assert np.isnan(out[H:3 * H]).all()
