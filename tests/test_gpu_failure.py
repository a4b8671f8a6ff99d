"""Failure detection on the GPU without a fault: each bounded device-side
wait of the library is made to run out (it waits on a flag, or an mbarrier,
that nothing sets, with a 50 ms limit); the kernel must record
STRIDE_DEV_TIMEOUT and return, and the context must stay usable (a normal
scoring call right after gives correct results).  Argument errors are
synchronous return codes (covered in test_gpu_batch.py)."""
import time

import numpy as np
import pytest

import synth
from gpu_helpers import LOGP_ATOL, run_batch

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("which", [0, 1], ids=["lookback_flag", "mbarrier"])
def test_bounded_wait_runs_out_and_reports(which):
    import torch

    import paper_2609_14636_gb300 as stride

    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(stride.stride_score_batch_workspace_size(2), dtype=torch.uint8, device="cuda")
    t0 = time.perf_counter()
    stride.stride_selftest_bounded_wait(which, 50_000_000, status, ws)
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    assert int(status.item()) & stride.DEV_TIMEOUT
    assert 0.04 <= dt < 5.0, dt
    # the context is still usable
    lay = synth.layout_from_turn_lengths([[3]])
    S = np.full((3, 64), 0x3F80, np.uint16)
    g = run_batch(stride, S, S, np.array([0, 1, 63], np.int32), lay, 1, -1e30)
    assert g["status"] == 0
    assert np.max(np.abs(g["logp_s"] + np.log(64.0))) <= LOGP_ATOL


def test_selftest_rejects_bad_arguments():
    import torch

    import paper_2609_14636_gb300 as stride

    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(stride.stride_score_batch_workspace_size(2), dtype=torch.uint8, device="cuda")
    with pytest.raises(stride.StrideError):
        stride.stride_selftest_bounded_wait(7, 1_000_000, status, ws)
    with pytest.raises(stride.StrideError):
        stride.stride_selftest_bounded_wait(0, 1_000_000, status, ws[:16])
