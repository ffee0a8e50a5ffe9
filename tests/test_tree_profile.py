"""The hardware-aware tree size helper (Section 4.2: Speedup(n) = tau(n) /
L_fp(n), pick the n that maximises it): tree shapes for every budget, the
speedup table and its argmax on CPU, and one latency profile on the GPU."""
import numpy as np
import pytest

from paper_2405_18628_gb300 import tree_profile
from paper_2405_18628_gb300 import workloads as W


@pytest.mark.parametrize("n", [1, 2, 3, 5, 16, 47, 64, 96, 127, 128])
def test_tree_size_workload_builds_n_token_trees(n):
    w = tree_profile.tree_size_workload(W.WORKLOADS["vicuna7b"], n)
    assert w.T == n and w.S_max == w.P + n
    rng = np.random.default_rng(n)
    parent, is_prompt = W.make_tree(rng, w)
    assert len(parent) == n and parent[0] == -1
    assert all(0 <= parent[i] < i for i in range(1, n))
    assert (~is_prompt).sum() == w.n_cand


def test_speedup_table_and_best_size():
    tau = {16: 2.0, 32: 2.6, 64: 3.0, 128: 3.1}
    lat = [(16, 1.0), (32, 1.1), (64, 1.4), (128, 2.5), (256, 5.0)]
    rows, best = tree_profile.speedup_table(tau, lat)
    assert [r["n"] for r in rows] == [16, 32, 64, 128]
    assert rows[1]["speedup"] == pytest.approx(2.6 / 1.1)
    assert best == 32
    # the rest of the forward pass shifts the optimum toward larger trees
    rows, best = tree_profile.speedup_table(tau, lat, extra_ms={n: 10.0 for n in tau})
    assert best == 64                     # 3.0 / 11.4 beats 2.6 / 11.1 and 3.1 / 12.5
    # ties: the smaller tree
    rows, best = tree_profile.speedup_table({8: 1.0, 16: 2.0}, [(8, 1.0), (16, 2.0)])
    assert best == 8
    assert tree_profile.speedup_table({}, lat) == ([], None)
    with pytest.raises(ValueError):
        tree_profile.speedup_table({16: 1.0}, [(16, 0.0)])


@pytest.mark.gpu
def test_latency_profile_on_gpu(cuda_device):
    base = W.scaled(W.WORKLOADS["mobilellama"], L=2, H=4)
    lat = tree_profile.latency_profile(base, [16, 64, 96], steps=5, warmup=2, device=cuda_device)
    assert [n for n, _ in lat] == [16, 64, 96]
    assert all(np.isfinite(ms) and ms > 0 for _, ms in lat)
