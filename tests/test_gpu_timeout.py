"""The device-side timeout, made to happen without faulting or hanging the GPU.

The one-grid step's CTAs wait for one another's argmax partials through flags
in the workspace, a wait bounded in time.  ppd_debug_grid_wait shortens the
bound to 1 ms and has one CTA withhold its flag, so every CTA's wait runs out:
the step must report PPD_ERR_TIMEOUT for every sequence and write no cache
row, and -- with the default bound restored and the workspace zeroed, as after
any timeout -- the next step on the same workspace must match the oracle.
The attention streams of the small case finish long before the 1 ms bound,
so only the grid-wide wait (a poll of global flags) gives up; no mbarrier or
TMA wait is made to expire."""
import numpy as np
import pytest
import torch

from paper_2405_18628_gb300 import ppd

from test_gpu_fused_modes import CASES, _check, _form, _inputs, _ref, _run

pytestmark = pytest.mark.gpu


def test_grid_wait_timeout_is_reported_and_recovered(cuda_device):
    w, pl = CASES["keyrow_200_v301"]          # 200 slices over a grid of one CTA per SM
    s, t = _inputs(w, pl)
    ref = _ref(s, t)
    ws = ppd.workspace(w.L, w.B, w.H, w.T, w.D, w.V, w.S_max, device=cuda_device)
    ws.zero_()
    prev = ppd.ppd_set_verify_step_form(2)
    try:
        assert _form(w) == 2
        ppd.ppd_debug_grid_wait(1_000_000, 1)  # 1 ms; CTA 1 never publishes its flag
        g, bufs = _run(w, s, t, cuda_device, ws=ws)
        np.testing.assert_array_equal(bufs.dev_status.cpu().numpy(),
                                      np.full(w.B, ppd.PPD_ERR_TIMEOUT, np.int32))
        for k in ("k_cache", "v_cache"):       # no accepted row was written
            assert torch.equal(g[k].cpu().view(torch.int16), t[k].view(torch.int16)), k
        ppd.ppd_debug_grid_wait(0, -1)
        ws.zero_()
        g2, bufs2 = _run(w, s, t, cuda_device, ws=ws)
        _check(w, s, t, g2, bufs2, ref, "the step after a timeout")
    finally:
        ppd.ppd_debug_grid_wait(0, -1)
        ppd.ppd_set_verify_step_form(prev)
