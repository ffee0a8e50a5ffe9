"""Host logic of bench.py: multi-rank runs (one replica per GPU, timing is the
slowest rank's), checked with two gloo ranks on the CPU, and the packed
buffers of the end-to-end leg."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        ms = 100.0 + 50.0 * rank                       # rank 1 is slower
        slowest = bench.max_over_ranks(ms, dist, "cpu")
        out[rank] = (slowest, bench.aggregate_rate(20, world, slowest))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_time():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(120)
            assert p.exitcode == 0
        res = dict(out)
    for r in range(world):
        slowest, rate = res[r]
        assert slowest == 150.0
        assert rate == pytest.approx(2 * 20 / 0.150)


def test_single_process_defaults():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.dist_setup({}) == (1, 0, 0)
    assert bench.dist_setup({"WORLD_SIZE": "4", "RANK": "2", "LOCAL_RANK": "2"}) == (4, 2, 2)
    assert bench.max_over_ranks(3.5) == 3.5
    assert bench.aggregate_rate(10, 1, 1000.0) == pytest.approx(10.0)


def test_packed_buffer_layout():
    """The end-to-end leg's one-copy buffers: every member at a 256-byte aligned
    offset, contiguous, with its own shape and dtype, and writable in place."""
    import torch
    sys.path.insert(0, ROOT)
    import bench
    buf, v = bench.packed({"q": ((2, 3, 5, 7), torch.bfloat16), "logits": ((3, 11), torch.float32),
                           "parent": ((4,), torch.int32)}, "cpu")
    for x in v.values():
        assert x.is_contiguous() and (x.data_ptr() - buf.data_ptr()) % 256 == 0
    assert v["q"].shape == (2, 3, 5, 7) and v["q"].dtype == torch.bfloat16
    assert v["logits"].dtype == torch.float32 and v["parent"].dtype == torch.int32
    assert buf.numel() == 512 + 256 + 256
    v["parent"].copy_(torch.arange(4, dtype=torch.int32))
    assert buf[768:784].view(torch.int32).tolist() == [0, 1, 2, 3]


def test_e2e_layer_groups():
    """The pipelined end-to-end leg's layer groups cover every layer once, the
    last group no larger than the first and the first no larger than the
    second."""
    sys.path.insert(0, ROOT)
    import bench
    for L in (1, 2, 4, 5, 6, 24, 32, 40, 80):
        g = bench.e2e_groups(L)
        assert sum(g) == L and all(n >= 1 for n in g)
        assert g[-1] <= g[0]
        assert len(g) == 1 or g[0] <= g[1]
    assert bench.e2e_groups(32) == [6, 8, 8, 6, 4]
