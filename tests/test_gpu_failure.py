"""Failure detection without a GPU fault: a bounded device-side wait on a barrier nothing arrives
on gives up, records SPD_ETIMEOUT in the workspace status word, and the context stays usable."""
import numpy as np
import pytest
import torch

from paper_2609_34977_gb300 import _native as N

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives():
    ws = torch.zeros(N.spd_linear_workspace_size(64, 128), dtype=torch.uint8, device="cuda")
    N.spd_selftest_bounded_wait(ws, 2_000_000)         # about a millisecond of SM clock
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == N.SPD_ETIMEOUT
    assert N.spd_workspace_status(ws) == N.SPD_OK       # reading clears the word
    X = torch.ones(64, 128, dtype=torch.bfloat16, device="cuda")
    W = torch.ones(128, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.empty(64, 128, device="cuda")
    N.spd_linear(X, 64, 128, W, 128, N.EPI_F32, out, 128, ws)
    torch.cuda.synchronize()
    assert torch.all(out == 128.0)


def test_host_side_rejections_touch_nothing():
    ws = torch.zeros(16, dtype=torch.uint8, device="cuda")
    X = torch.ones(4, 128, dtype=torch.bfloat16, device="cuda")
    W = torch.ones(128, 128, dtype=torch.bfloat16, device="cuda")
    out = torch.zeros(4, 128, device="cuda")
    with pytest.raises(N.SpiderError) as e:
        N.spd_linear(X, 4, 128, W, 128, N.EPI_F32, out, 128, ws)   # workspace too small
    assert e.value.code == N.SPD_ENOSPC
    with pytest.raises(ValueError):                                 # weights too small (binding)
        N.spd_linear(X, 4, 128, X, 128, N.EPI_F32, out, 128, ws)
    torch.cuda.synchronize()
    assert not out.any()
