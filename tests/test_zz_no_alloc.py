"""spd_linear_noalloc (the workspace-free spd_linear, scratch in a static device array of the
library) against spd_linear on the same operands, through the C ABI. Kept in its own file, named
to be collected last, so it runs both alone in a fresh process (its first call then does the
per-device set-up) and after every other GPU test.

Tolerances are those of the GEMM tests: fp32 outputs within 1e-4 of each row's magnitude, bf16
outputs within 1e-2 (one bf16 rounding)."""
import numpy as np
import pytest
import torch

from paper_2609_34977_gb300 import _native as N
from tests.gpu_util import bf16_np, rowwise_rel

pytestmark = pytest.mark.gpu


def operands(M, K, N_, seed):
    g = torch.Generator().manual_seed(seed)
    X = torch.randn(M, K, generator=g).to(torch.bfloat16).cuda()
    W = (torch.randn(N_, K, generator=g) * 0.05).to(torch.bfloat16).cuda()
    bias = (torch.randn(N_, generator=g) * 0.1).to(torch.bfloat16).cuda()
    return X, W, bias


@pytest.mark.parametrize("M,K,N_,epi", [
    (300, 1024, 640, N.EPI_F32),           # stream-K with split tiles (partial slots in the scratch)
    (256, 4096, 4096, N.EPI_F32),          # cluster split-K (no partial slots)
    (70, 1024, 384, N.EPI_BIAS_GELU_BF16),  # bf16 epilogue with bias
    (8, 4096, 1000, N.EPI_F32),            # tiny token count: 256-row weight tiles, ragged N
])
def test_noalloc_matches_workspace_entry_on_two_calls(M, K, N_, epi):
    X, W, bias = operands(M, K, N_, seed=M + N_)
    f32 = epi == N.EPI_F32
    dt = torch.float32 if f32 else torch.bfloat16
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    ref = torch.zeros(M, N_, dtype=dt, device="cuda")
    N.spd_linear(X, M, K, W, N_, epi, ref, N_, ws, bias=bias)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    ref = ref.float().cpu().numpy() if f32 else bf16_np(ref)
    tol = 1e-4 if f32 else 1e-2
    status = torch.full((1,), -99, dtype=torch.int32, device="cuda")
    for _ in range(2):
        out = torch.full((M, N_), float("nan"), dtype=dt, device="cuda")
        N.spd_linear_noalloc(X, M, K, W, N_, epi, out, N_, bias=bias, status=status)
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        got = out.float().cpu().numpy() if f32 else bf16_np(out)
        assert np.isfinite(got).all()
        assert rowwise_rel(got, ref) < tol


def test_noalloc_residual_add_into_rows():
    M, K, N_ = 90, 2048, 512
    X, W, _ = operands(M, K, N_, seed=3)
    h0 = torch.randn(200, N_, device="cuda")
    rows = torch.randperm(200)[:M].to(torch.int32).cuda()
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    ref = h0.clone()
    N.spd_linear(X, M, K, W, N_, N.EPI_ADD_F32, ref, N_, ws, rows=rows)
    for _ in range(2):
        h = h0.clone()
        N.spd_linear_noalloc(X, M, K, W, N_, N.EPI_ADD_F32, h, N_, rows=rows)
        torch.cuda.synchronize()
        assert rowwise_rel(h.cpu().numpy(), ref.cpu().numpy()) < 1e-4


@pytest.mark.parametrize("M,N_", [
    (1, 4097 * 128),  # 2 x 2049 counters for one token tile
    (600, 1365 * 128),  # 2 x 683 x 3 = 4098 counters (CTA pairs count each half of a 256-row tile)
])
def test_noalloc_rejects_problems_beyond_its_scratch(M, N_):
    # more tile counters than the static scratch holds: refused on the host, nothing enqueued
    K = 64
    X = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(N_, K, dtype=torch.bfloat16, device="cuda")  # never read
    out = torch.zeros(M, N_, dtype=torch.float32, device="cuda")  # never written
    with pytest.raises(N.SpiderError) as e:
        N.spd_linear_noalloc(X, M, K, W, N_, N.EPI_F32, out, N_)
    assert e.value.code == N.SPD_ENOSPC
    torch.cuda.synchronize()
    assert not out.any()
