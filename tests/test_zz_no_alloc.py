"""ppd_node_argmax_noalloc: the node argmax for callers that cannot allocate
device memory (a plugin handed only its input and output tensors, a loop that
forbids allocation after start-up, a fixed memory budget).  Its partial maxima
live in a fixed array inside the library instead of a caller workspace.

The results must equal the fp64 oracle's argmax and ppd_node_argmax's bit for
bit, on consecutive calls that reuse the shared array with different shapes
(up to the largest request the array holds, B*T = 65,536 node rows, with
16-byte and scalar loads), and oversized requests must be refused before any
work is enqueued.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle

pytestmark = pytest.mark.gpu


def _logits(B, T, V, seed):
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((B, T, V)).astype(np.float32)
    flat = x.reshape(B * T, V)
    flat[0, [3, V - 2]] = 99.0                  # tie: the lower index wins
    if B * T > 1:
        flat[1, [V // 2, 5]] = np.nan           # first NaN wins
    if B * T > 2:
        flat[2, :] = -np.inf                    # all equal: index 0
    if B * T > 3:
        flat[3, :] = -1.0
        flat[3, [V - 1, 1]] = [0.0, -0.0]       # -0 == +0: the lower index
    if B * T > 100:
        # ties between neighbouring rows' extremes and in the last column
        flat[100:, V - 1] = flat[100:].max(axis=1)
    return x


@pytest.mark.parametrize("shapes", [[(2, 64, 32000), (1, 7, 1001), (1, 65536, 16),
                                     (1, 65536, 18)]])
def test_noalloc_argmax_matches_oracle_and_workspace_argmax(cuda_device, shapes):
    from paper_2405_18628_gb300 import ppd
    for call, (B, T, V) in enumerate(shapes):            # consecutive calls, shapes change
        xh = _logits(B, T, V, seed=call)
        want = oracle.node_argmax(xh)
        x = torch.from_numpy(xh).to(cuda_device)
        ref = torch.full((B, T), -1, dtype=torch.int32, device=cuda_device)
        ws = ppd.workspace(1, B, 1, T, 64, V, 1, device=cuda_device)
        ppd.ppd_node_argmax(x, ref, ws)
        got = torch.full((B, T), -2, dtype=torch.int32, device=cuda_device)
        ppd.ppd_node_argmax_noalloc(x, got)
        torch.cuda.synchronize()
        g = got.cpu().numpy()
        np.testing.assert_array_equal(g, want, err_msg=f"call {call} {B}x{T}x{V} vs oracle")
        assert torch.equal(got, ref), f"call {call}: differs from ppd_node_argmax"


def test_noalloc_argmax_rejects_too_many_rows(cuda_device):
    from paper_2405_18628_gb300 import ppd
    lib = ppd.load()
    fake = ctypes.c_void_p(0x10000)            # never touched: the size check fails first
    st = lib.ppd_node_argmax_noalloc(fake, 2, 32769, 16, fake, ctypes.c_void_p(0))
    assert st == ppd.PPD_ERR_UNSUPPORTED
    assert lib.ppd_node_argmax_noalloc(fake, 1, 65536, 16, None, ctypes.c_void_p(0)) == \
        ppd.PPD_ERR_INVALID_ARG
