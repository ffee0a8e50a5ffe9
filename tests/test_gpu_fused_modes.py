"""The fused verification step computes the node argmax either in a grid of its
own ahead of the attention grid (form 1), or inside the attention grid, where
the spare warp of every CTA takes a share of the (row, split) chunks while the
K/V stream runs and the CTAs exchange per-call flags tagged with an epoch kept
in the workspace (form 2).  These tests pin the in-grid form, forced through
ppd_set_verify_step_form where the automatic choice would differ, against the
fp64 oracle -- indices, paths, statuses and compacted KV bit for bit,
attention within tolerance -- over every kernel layout, several sequences with
their own prefixes, batches up to 64, junk workspaces, calls back to back, and
CUDA-graph replays; and the argmax grid, at the widths the step launches it
with, the same way."""
import numpy as np
import pytest
import torch

import oracle
from paper_2405_18628_gb300 import ppd
from paper_2405_18628_gb300 import workloads as W

from test_gpu_parity import assert_attn_close, i32, tensors
from test_gpu_typical import DELTA, EPS, TEMP, _margins_clear

pytestmark = pytest.mark.gpu


def in_grid(w):
    """The library's choice of mode (in_grid_argmax_pays in ppd_api.cu): in-grid
    when 64 x the logits bytes are at most the K/V bytes over S_max + T rows."""
    return 4 * w.B * w.T * w.V * 64 <= 4 * w.L * w.B * w.H * (w.S_max + w.T) * w.D


def _wl(name, seed, **kw):
    base = dict(n_cand=12, max_depth=4, chains="fill3", match_rate=0.7, seed=seed)
    base.update(kw)
    return W.Workload(name, **base)


CASES = {
    # key-row kernel, work split (24 slices), scalar logits loads (V % 4 != 0)
    "keyrow_split_v301": (_wl("a", 501, L=2, B=3, H=4, D=64, P=1500, T=40, V=301),
                          [1500, 700, 3]),
    # key-row kernel, whole slices round-robin (256 slices)
    "keyrow_roundrobin": (_wl("b", 502, L=4, B=2, H=32, D=64, P=600, T=32, V=512), [600, 411]),
    # query-row kernel, one block of 128 queries
    "rows_t100": (_wl("c", 503, L=1, B=2, H=4, D=128, P=3000, T=100, V=248, n_cand=30),
                  [3000, 2048]),
    # query-row kernel, three query blocks
    "rows_t285": (_wl("d", 504, L=1, B=1, H=8, D=128, P=3000, T=285, V=192, n_cand=72),
                  [2999]),
    # the largest fused batch
    "batch64": (_wl("e", 505, L=1, B=64, H=2, D=64, P=1000, T=16, V=120, n_cand=8, max_depth=3,
                    chains="every1"), None),
    # 200 slices over 152 SMs (a partial second round); scalar loads (V % 4 != 0)
    "keyrow_200_v301": (_wl("g", 507, L=1, B=2, H=100, D=64, P=1500, T=40, V=301),
                        [1500, 777]),
    # key-row kernel with D = 128 and 16-byte loads
    "keyrow_200_d128": (_wl("h", 508, L=2, B=1, H=100, D=128, P=700, T=64, V=1000, n_cand=20),
                        [700]),
    # query-row kernel, 200 slices
    "rows_200_t100": (_wl("i", 509, L=1, B=2, H=100, D=128, P=900, T=100, V=248, n_cand=30),
                      [900, 300]),
}


def _form(w):
    return ppd.ppd_verify_step_form(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max)


@pytest.fixture
def form():
    """Force the in-grid form for one test, then restore the automatic choice."""
    prev = ppd.ppd_set_verify_step_form(2)
    yield 2
    ppd.ppd_set_verify_step_form(prev)


def _inputs(w, pl, seed=None):
    if pl is None:
        pl = np.random.default_rng(w.seed).integers(0, w.P + 1, size=w.B)
    s = W.make_step_inputs(w, seed=seed, prefix_len=np.asarray(pl, np.int32))
    t = tensors(w, seed=seed, prefix_len=s.prefix_len)
    return s, t


def _run(w, s, t, dev, ws=None, typical=False):
    g = {k: v.to(dev) for k, v in t.items()}
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev, with_lse=True)
    for k in ("argmax", "accept_len", "path", "next_token", "new_prefix_len", "dev_status"):
        getattr(bufs, k).fill_(-99)
    wsp = bufs.workspace if ws is None else ws
    args = (g["q"], g["k_cache"], g["v_cache"], g["k_tree"], g["v_tree"], i32(s.prefix_len, dev),
            i32(s.parent, dev), i32(s.cand_tokens, dev), torch.from_numpy(s.logits).to(dev))
    outs = (bufs.out, bufs.argmax, bufs.accept_len, bufs.path, bufs.next_token,
            bufs.new_prefix_len, bufs.dev_status, wsp)
    if typical:
        ppd.ppd_verify_step_typical(*args, TEMP, EPS, DELTA, *outs, lse=bufs.lse)
    else:
        ppd.ppd_verify_step(*args, *outs, lse=bufs.lse)
    torch.cuda.synchronize()
    return g, bufs


def _check(w, s, t, g, bufs, ref, what):
    assert_attn_close(bufs.out.cpu().numpy().reshape(ref["out"].shape), ref["out"], what)
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), ref["argmax"], err_msg=what)
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=f"{what} {k}")
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), ref["status"], err_msg=what)
    for k in ("k_cache", "v_cache"):
        np.testing.assert_array_equal(g[k].cpu().view(torch.int16).numpy().view(np.uint16), ref[k],
                                      err_msg=f"{what} {k}")


def _ref(s, t):
    return oracle.verify_step(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                              s.prefix_len, s.parent, s.cand_tokens, s.logits)


@pytest.mark.parametrize("case", sorted(CASES))
def test_in_grid_step_matches_oracle(cuda_device, case, form):
    w, pl = CASES[case]
    assert _form(w) == form
    s, t = _inputs(w, pl)
    ref = _ref(s, t)
    g, bufs = _run(w, s, t, cuda_device)
    _check(w, s, t, g, bufs, ref, case)
    assert (ref["accept_len"] >= 1).all()


@pytest.mark.parametrize("case", ["keyrow_split_v301", "keyrow_200_v301"])
def test_in_grid_typical_step_matches_oracle(cuda_device, case, form):
    w, pl = CASES[case]
    s, t = _inputs(w, pl, seed=77)
    ref = oracle.verify_step_typical(t["q"], t["k_cache"], t["v_cache"], t["k_tree"], t["v_tree"],
                                     s.prefix_len, s.parent, s.cand_tokens, s.logits, TEMP, EPS,
                                     DELTA)
    assert _margins_clear(ref)
    g, bufs = _run(w, s, t, cuda_device, typical=True)
    _check(w, s, t, g, bufs, ref, "typical in-grid")


@pytest.mark.parametrize("case", ["keyrow_split_v301", "keyrow_200_d128"])
def test_in_grid_junk_workspace(cuda_device, case, form):
    """Whatever the workspace holds (flags and epoch included), two calls in a
    row give the oracle's results: each call tags its flags with a fresh epoch."""
    w, pl = CASES[case]
    s, t = _inputs(w, pl)
    ref = _ref(s, t)
    ws = ppd.workspace(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=cuda_device)
    gen = torch.Generator(device="cpu").manual_seed(3)
    fills = [0xFF, 0x7F, 0x00, None]
    for fill in fills:
        if fill is None:
            ws.copy_(torch.randint(0, 256, ws.shape, dtype=torch.uint8, generator=gen))
        else:
            ws.fill_(fill)
        for rep in range(2):
            g, bufs = _run(w, s, t, cuda_device, ws=ws)
            _check(w, s, t, g, bufs, ref, f"fill {fill} call {rep}")


def test_in_grid_workspace_reused_across_shapes(cuda_device, form):
    """One workspace (sized for the largest) serving in-grid steps of different
    shapes in turn: the epoch word and flags stay at the workspace's start for
    every shape, so no call sees stale flags of another shape's layout."""
    names = ["rows_t285", "keyrow_roundrobin", "batch64", "keyrow_split_v301", "rows_t285"]
    n = max(ppd.ppd_workspace_bytes(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max)
            for w, _ in (CASES[k] for k in names))
    ws = torch.zeros(n, dtype=torch.uint8, device=cuda_device)
    for i, name in enumerate(names):
        w, pl = CASES[name]
        s, t = _inputs(w, pl)
        g, bufs = _run(w, s, t, cuda_device, ws=ws)
        _check(w, s, t, g, bufs, _ref(s, t), f"{name} (call {i})")


def test_in_grid_calls_back_to_back(cuda_device, form):
    """Different steps through one workspace, enqueued without host syncs in
    between: each sees only its own argmax partials."""
    w, pl = CASES["keyrow_roundrobin"]
    ws = ppd.workspace(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=cuda_device)
    dev = cuda_device
    runs = []
    for seed in (11, 12, 13, 14):
        s, t = _inputs(w, pl, seed=seed)
        g = {k: v.to(dev) for k, v in t.items()}
        bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
        ppd.ppd_verify_step(g["q"], g["k_cache"], g["v_cache"], g["k_tree"], g["v_tree"],
                            i32(s.prefix_len, dev), i32(s.parent, dev), i32(s.cand_tokens, dev),
                            torch.from_numpy(s.logits).to(dev), bufs.out, bufs.argmax,
                            bufs.accept_len, bufs.path, bufs.next_token, bufs.new_prefix_len,
                            bufs.dev_status, ws)
        runs.append((s, t, g, bufs))
    torch.cuda.synchronize()
    for i, (s, t, g, bufs) in enumerate(runs):
        _check(w, s, t, g, bufs, _ref(s, t), f"call {i}")


def test_in_grid_graph_replays(cuda_device, form):
    """The step captured once in a CUDA graph and replayed with a new tree,
    candidates and logits each time: the epoch advances on the device, so
    every replay gets fresh flags."""
    w, pl = CASES["rows_t100"]
    dev = cuda_device
    s, t = _inputs(w, pl, seed=21)
    g = {k: v.to(dev) for k, v in t.items()}
    pre, par, cand = i32(s.prefix_len, dev), i32(s.parent, dev), i32(s.cand_tokens, dev)
    logits = torch.from_numpy(s.logits).to(dev)
    bufs = ppd.StepBuffers(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=dev)
    side = torch.cuda.Stream()

    def step():
        ppd.ppd_verify_step(g["q"], g["k_cache"], g["v_cache"], g["k_tree"], g["v_tree"], pre, par,
                            cand, logits, bufs.out, bufs.argmax, bufs.accept_len, bufs.path,
                            bufs.next_token, bufs.new_prefix_len, bufs.dev_status, bufs.workspace,
                            stream=side)

    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()                                   # warm-up outside the capture
    side.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=side):
        step()
    for seed in (31, 32, 33):
        s2 = W.make_step_inputs(w, seed=seed, prefix_len=s.prefix_len)
        par.copy_(i32(s2.parent, dev))
        cand.copy_(i32(s2.cand_tokens, dev))
        logits.copy_(torch.from_numpy(s2.logits))
        for k in ("k_cache", "v_cache"):
            g[k].copy_(t[k])
        graph.replay()
        torch.cuda.synchronize()
        _check(w, s2, t, g, bufs, _ref(s2, t), f"replay seed {seed}")


@pytest.mark.parametrize("fused_form", [1, 2])
def test_in_grid_argmax_ties_nans_and_chunk_edges(cuda_device, fused_form):
    """Both argmax forms follow the library's ranking rule (first NaN, then the
    largest value, then the lowest index; -0 == +0) across the boundaries of
    the column chunks (2048 logits at V = 8192 and 32 rows; 256 slices on 152
    SMs, so form 1 runs its narrow argmax grid on the idle SMs of the second
    round), bit for bit against the oracle, and the step's acceptance with it."""
    w = _wl("f", 506, L=4, B=2, H=32, D=64, P=4000, T=16, V=8192, n_cand=8, chains="every1")
    prev = ppd.ppd_set_verify_step_form(fused_form)
    try:
        _ties_case(cuda_device, w, fused_form)
    finally:
        ppd.ppd_set_verify_step_form(prev)


def _ties_case(cuda_device, w, form):
    assert _form(w) == form
    s, t = _inputs(w, [w.P, 1234])
    x = s.logits
    x[0, 1, :] = -1.0
    x[0, 1, 2047] = x[0, 1, 2048] = 5.0            # tie straddling side chunks 0 and 1
    x[0, 2, 5000] = np.nan
    x[0, 2, 7000] = np.nan                          # first NaN wins, in a later chunk
    x[0, 3, :] = -np.inf                            # all -inf: index 0
    x[0, 4, 6000] = x[0, 4, 6001] = np.inf          # +inf tie inside one chunk
    x[0, 5, :] = 0.25                               # constant row: index 0
    x[0, 6, :] = -3.0
    x[0, 6, 4096] = -0.0
    x[0, 6, 4095] = 0.0                             # -0 == +0: the lower index
    x[0, 7, :] = -1.0
    x[0, 7, 6143] = x[0, 7, 6144] = 9.0             # tie straddling chunks 2 and 3
    x[0, 8, 4096] = np.nan
    x[0, 8, 4095] = np.nan                          # NaNs either side of chunks 1 | 2
    x[0, 9, :] = -5.0
    x[0, 9, [7167, 2048, 6144]] = 2.5               # three-way tie over three chunks
    x[1, 0, :] = -2.0
    x[1, 0, 8191] = 7.0                             # the very last logit
    x[1, 1, :] = np.nan                             # all NaN: index 0
    ref = _ref(s, t)
    assert ref["argmax"][0, 1] == 2047 and ref["argmax"][0, 2] == 5000
    assert ref["argmax"][0, 6] == 4095 and ref["argmax"][1, 0] == 8191
    assert ref["argmax"][0, 7] == 6143 and ref["argmax"][0, 8] == 4095
    assert ref["argmax"][0, 9] == 2048
    g, bufs = _run(w, s, t, cuda_device)
    np.testing.assert_array_equal(bufs.argmax.cpu().numpy(), ref["argmax"])
    _check(w, s, t, g, bufs, ref, f"ties and NaNs, form {form}")


@pytest.mark.parametrize("case", ["keyrow_split_v301", "keyrow_200_v301"])
def test_in_grid_reports_bad_sequences(cuda_device, case, form):
    """Per-sequence status in the in-grid form, written by each sequence's
    designated CTA: a malformed tree and (three sequences) a prefix with no
    room left."""
    w, pl = CASES[case]
    s, t = _inputs(w, pl)
    s.parent[1, 7] = 9
    if w.B > 2:
        s.prefix_len[2] = w.S_max
    t = tensors(w, prefix_len=s.prefix_len)
    ref = _ref(s, t)
    assert ref["status"].tolist() == [0, 3, 4][:w.B]
    g, bufs = _run(w, s, t, cuda_device)
    # attention outputs of a failed sequence are unspecified: indices, statuses
    # and the cache only
    np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(), ref["status"])
    for k in ("accept_len", "path", "next_token", "new_prefix_len"):
        np.testing.assert_array_equal(getattr(bufs, k).cpu().numpy(), ref[k], err_msg=k)
    for k in ("k_cache", "v_cache"):
        np.testing.assert_array_equal(g[k].cpu().view(torch.int16).numpy().view(np.uint16), ref[k],
                                      err_msg=k)


@pytest.mark.parametrize("typical", [False, True], ids=["exact", "typical"])
@pytest.mark.parametrize("case", ["keyrow_roundrobin", "keyrow_200_v301", "rows_200_t100",
                                  "keyrow_split_v301"])
def test_argmax_grid_form(cuda_device, case, typical):
    """Form 1 (an argmax grid, then the attention grid) against the oracle: on
    the idle SMs of a partial round of slices the step runs a narrow argmax
    grid (the first three cases), under the work split the wide one (the
    last).  Exact matching and typical acceptance."""
    w, pl = CASES[case]
    s, t = _inputs(w, pl)
    prev = ppd.ppd_set_verify_step_form(1)
    try:
        assert _form(w) == 1
        if typical:
            ref = oracle.verify_step_typical(t["q"], t["k_cache"], t["v_cache"], t["k_tree"],
                                             t["v_tree"], s.prefix_len, s.parent, s.cand_tokens,
                                             s.logits, TEMP, EPS, DELTA)
            assert _margins_clear(ref)
        else:
            ref = _ref(s, t)
        g, bufs = _run(w, s, t, cuda_device, typical=typical)
    finally:
        ppd.ppd_set_verify_step_form(prev)
    _check(w, s, t, g, bufs, ref, f"{case} form 1")
