"""The C-ABI library: it builds, loads, exports every entry point that
include/ppd.h declares, and rejects bad arguments on the host before any
device work (no GPU needed: these calls return before touching CUDA)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2405_18628_gb300 import build, ppd
    build.build()
    return ppd.load()


def _declared():
    src = open(os.path.join(ROOT, "include", "ppd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ppd_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("ppd_tree_attention", "ppd_node_argmax", "ppd_accept_path", "ppd_kv_compact",
              "ppd_verify_step", "ppd_workspace_bytes", "ppd_status_string"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared():
        assert hasattr(lib, name), name


def test_status_strings(lib):
    from paper_2405_18628_gb300 import ppd
    for s in range(7):
        assert ppd.status_string(s) and ppd.status_string(s) != "unknown status"
    assert ppd.status_string(99) == "unknown status"


def test_workspace_bytes(lib):
    from paper_2405_18628_gb300 import ppd
    a = ppd.ppd_workspace_bytes(32, 1, 32, 64, 128, 32000, 2112)
    assert a > 0 and a % 256 == 0
    f = ppd.ppd_workspace_bytes(1, 1, 4, 48, 64, 1024, 176, ppd.PPD_F32)
    assert f >= 2 * (3 * 48 + 2 * 176) * 64 * 4
    assert ppd.ppd_workspace_bytes(0, 1, 1, 1, 64, 1, 1) == 0


def test_verify_step_launch_counts(lib):
    """Kernels per verification step: a one-block status reset and one grid
    when the argmax runs inside the attention grid (Vicuna-7B shapes on a
    device of unknown SM count: 8 MB of logits against 1.1 GB of K/V), an
    argmax grid first when the logits weigh more (48 x 1024 logits against a
    128-token prefix), five grids above 64 sequences, five fp32 rounding grids
    in front for fp32 operands, and -1 for sizes the step rejects."""
    from paper_2405_18628_gb300 import ppd
    assert ppd.ppd_verify_step_launches(32, 1, 32, 64, 128, 32000, 2112) == 2
    assert ppd.ppd_verify_step_launches(32, 1, 32, 64, 128, 32000, 2112, typical=True) == 2
    assert ppd.ppd_verify_step_launches(1, 1, 4, 48, 64, 1024, 176) == 2
    assert ppd.ppd_verify_step_launches(1, 1, 4, 48, 64, 1024, 176, ppd.PPD_F32) == 7
    assert ppd.ppd_verify_step_launches(1, 65, 2, 16, 64, 300, 56) == 5
    assert ppd.ppd_verify_step_launches(1, 1, 4, 48, 96, 1024, 176) == -1
    assert ppd.ppd_verify_step_launches(1, 1, 4, 48, 64, 0, 176) == -1


def test_verify_step_forms(lib):
    """The fused step's form: separate grids above 64 sequences, an argmax grid
    first when the logits weigh more than 1/64 of the K/V bytes (the tiny
    shapes) or when a narrow argmax grid fits the SMs left idle by the last
    round of slices (the Vicuna-7B shapes on 152 SMs), the argmax in the
    attention grid's side warps otherwise, -1 for rejected sizes.  The
    side-warp case uses 171 layers of the Vicuna-7B shapes: 5472 slices leave
    fewer than 8 SMs of the last round idle on 148 SMs (the count assumed
    without a GPU) and none on 152.  A forced form applies to every fused size
    until it is reset, and other values are refused."""
    from paper_2405_18628_gb300 import ppd
    assert ppd.ppd_verify_step_form(1, 65, 2, 16, 64, 300, 56) == 0
    assert ppd.ppd_verify_step_form(1, 1, 4, 48, 64, 1024, 176) == 1
    assert ppd.ppd_verify_step_form(171, 1, 32, 64, 128, 32000, 2112) == 2
    assert ppd.ppd_verify_step_form(32, 1, 32, 64, 128, 32000, 2112) in (1, 2)
    assert ppd.ppd_verify_step_form(1, 1, 4, 48, 96, 1024, 176) == -1
    prev = ppd.ppd_set_verify_step_form(2)
    try:
        assert prev == -1
        assert ppd.ppd_verify_step_form(1, 1, 4, 48, 64, 1024, 176) == 2
        assert ppd.ppd_verify_step_form(1, 65, 2, 16, 64, 300, 56) == 0
        assert ppd.ppd_verify_step_launches(1, 1, 4, 48, 64, 1024, 176) == 2
        assert ppd.ppd_set_verify_step_form(1) == 2
        assert ppd.ppd_verify_step_launches(32, 1, 32, 64, 128, 32000, 2112) == 2
        for bad in (0, 3, 4):
            assert ppd.ppd_set_verify_step_form(bad) == -2
        assert ppd.ppd_verify_step_form(1, 1, 4, 48, 64, 1024, 176) == 1
    finally:
        ppd.ppd_set_verify_step_form(-1)
    assert ppd.ppd_verify_step_form(171, 1, 32, 64, 128, 32000, 2112) == 2


def test_host_argument_checks(lib):
    """Invalid sizes and null pointers are rejected with PPD_ERR_INVALID_ARG
    (or UNSUPPORTED) without launching anything."""
    vp = ctypes.c_void_p
    fake = vp(0x10000)            # never dereferenced: the checks fail first
    null = None
    s = vp(0)
    INVALID = 1
    # the timeout diagnostics reject a negative CTA other than -1, and restore cleanly
    assert lib.ppd_debug_grid_wait(ctypes.c_ulonglong(0), -2) == INVALID
    assert lib.ppd_debug_grid_wait(ctypes.c_ulonglong(0), -1) == 0
    # T > 512
    assert lib.ppd_tree_attention(fake, fake, fake, fake, fake, fake, fake, 1, 1, 1, 513, 64, 200,
                                  0, 0.0, fake, null, fake, null, 0, s) == INVALID
    # D not in {64, 128}
    assert lib.ppd_tree_attention(fake, fake, fake, fake, fake, fake, fake, 1, 1, 1, 8, 96, 200,
                                  0, 0.0, fake, null, fake, null, 0, s) == INVALID
    # null output
    assert lib.ppd_tree_attention(fake, fake, fake, fake, fake, fake, fake, 1, 1, 1, 8, 64, 200,
                                  0, 0.0, null, null, fake, null, 0, s) == INVALID
    # misaligned q
    assert lib.ppd_tree_attention(vp(0x10002), fake, fake, fake, fake, fake, fake, 1, 1, 1, 8, 64,
                                  200, 0, 0.0, fake, null, fake, null, 0, s) == INVALID
    # fp32 without workspace
    assert lib.ppd_tree_attention(fake, fake, fake, fake, fake, fake, fake, 1, 1, 1, 8, 64, 200,
                                  1, 0.0, fake, null, fake, null, 0, s) == INVALID
    assert lib.ppd_node_argmax(fake, 0, 4, 10, fake, null, 0, s) == INVALID
    assert lib.ppd_node_argmax(fake, 1, 64, 32000, fake, null, 0, s) == INVALID   # needs workspace
    assert lib.ppd_accept_path(fake, fake, fake, fake, 1, 600, 10, 10, fake, fake, fake, fake,
                               fake, s) == INVALID
    assert lib.ppd_accept_path(fake, fake, null, fake, 1, 4, 10, 10, fake, fake, fake, fake,
                               fake, s) == INVALID
    # compaction: tree buffer inside the cache buffer
    assert lib.ppd_kv_compact(vp(0x100000), vp(0x900000), vp(0x100400), vp(0xA00000), fake, fake,
                              fake, 1, 1, 1, 4, 64, 100, 0, s) == INVALID
    # verify step: missing workspace
    args = [fake] * 9 + [1, 1, 1, 8, 64, 100, 200, 0, 0.0] + [fake] * 8 + [null, 0, s]
    assert lib.ppd_verify_step(*args) == INVALID


def test_binding_requires_library(monkeypatch, tmp_path):
    from paper_2405_18628_gb300 import ppd
    monkeypatch.setattr(ppd, "_lib", None)
    monkeypatch.setattr(ppd, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="missing"):
        ppd.load()


def test_typical_acceptance_host_checks(lib):
    """Typical acceptance needs a positive, finite temperature and finite
    epsilon / delta; bad values are refused before any launch."""
    from paper_2405_18628_gb300 import ppd
    vp = ctypes.c_void_p
    fake = vp(0x10000)
    s = vp(0)
    ws = 1 << 20
    for temp in (0.0, -1.0, float("nan"), float("inf"), 1e-45):
        assert lib.ppd_node_stats(fake, 1, 4, 100, temp, fake, fake, fake, fake, ws, s) == \
            ppd.PPD_ERR_INVALID_ARG
        assert lib.ppd_typical_accept(*[fake] * 7, 1, 4, 100, 10, temp, 0.1, 0.1,
                                      *[fake] * 5, s) == ppd.PPD_ERR_INVALID_ARG
    for eps, delta in ((float("nan"), 0.1), (0.1, float("inf"))):
        assert lib.ppd_typical_accept(*[fake] * 7, 1, 4, 100, 10, 1.0, eps, delta,
                                      *[fake] * 5, s) == ppd.PPD_ERR_INVALID_ARG
    args = [fake] * 9 + [1, 1, 1, 4, 64, 100, 16, ppd.PPD_BF16, 0.0, 0.0, 0.1, 0.1] + \
        [fake] * 8 + [fake, 1 << 30, s]
    assert lib.ppd_verify_step_typical(*args) == ppd.PPD_ERR_INVALID_ARG
    assert lib.ppd_node_stats(None, 1, 4, 100, 1.0, fake, fake, fake, fake, ws, s) == \
        ppd.PPD_ERR_INVALID_ARG


def test_next_tree_host_checks(lib):
    """Next-step tree: K in 1..16 and <= V, n_ept in 1..128, n_states <= 128,
    T and T_next <= 512, enough workspace; refused before any launch."""
    from paper_2405_18628_gb300 import ppd
    vp = ctypes.c_void_p
    fake = vp(0x10000)
    s = vp(0)
    ws = 1 << 20

    def call(B=2, T=16, V=100, n_states=4, T_next=32, K=4, n_ept=1, ws_bytes=ws):
        return lib.ppd_next_tree(*[fake] * 6, B, T, V, n_states, T_next, fake, fake, K, n_ept,
                                 *[fake] * 4, fake, ws_bytes, s)

    assert call(n_ept=0) == ppd.PPD_ERR_INVALID_ARG
    assert call(n_ept=129) == ppd.PPD_ERR_UNSUPPORTED
    assert call(K=17) == ppd.PPD_ERR_UNSUPPORTED
    assert call(K=0) == ppd.PPD_ERR_INVALID_ARG
    assert call(K=8, V=7) == ppd.PPD_ERR_INVALID_ARG
    assert call(n_states=129) == ppd.PPD_ERR_INVALID_ARG
    assert call(T=513) == ppd.PPD_ERR_INVALID_ARG
    assert call(T_next=513) == ppd.PPD_ERR_INVALID_ARG
    need = lib.ppd_next_tree_workspace_bytes(2, 4, 4)
    assert need >= 2 * 4 * 4 * 4 + 2 * 4
    assert call(ws_bytes=need - 1) == ppd.PPD_ERR_INVALID_ARG

    def call_ept(ept_mean, n_ept=2, K=4):
        return lib.ppd_next_tree_ept(*[fake] * 6, 2, 16, 100, 4, 32, fake, fake, K, n_ept,
                                     ept_mean, *[fake] * 4, fake, ws, s)

    assert call_ept(2) == ppd.PPD_ERR_INVALID_ARG
    assert call_ept(-1) == ppd.PPD_ERR_INVALID_ARG
    assert call_ept(1, n_ept=129) == ppd.PPD_ERR_UNSUPPORTED
    assert call_ept(1, K=17) == ppd.PPD_ERR_UNSUPPORTED
