"""tcgen05 GEMM (spd_linear) against the plain definition out = X W^T (fp64 on the CPU from the
same bf16 operands). fp32 accumulation: tolerance 1e-4 of each output row's magnitude."""
import numpy as np
import pytest
import torch

from paper_2609_34977_gb300 import _native as N
from tests.gpu_util import bf16_np, rowwise_rel

pytestmark = pytest.mark.gpu


def operands(M, K, N_, seed=0):
    g = torch.Generator().manual_seed(seed)
    X = torch.randn(M, K, generator=g).to(torch.bfloat16)
    W = (torch.randn(N_, K, generator=g) * 0.05).to(torch.bfloat16)
    return X, W


@pytest.mark.parametrize("M,K,N_", [
    (1, 64, 128), (20, 256, 256), (64, 688, 384), (128, 1024, 512), (100, 4096, 256),
    (256, 4096, 4096),          # split-K path (few tiles)
    (300, 512, 1024),           # two token tiles with a ragged tail
    (640, 1024, 640),           # dense LLaVA row count, three token tiles
    (37, 11008, 384),           # K = d_ffn, long split-K
    (8, 4096, 1000),            # N not a multiple of 128 (LM-head-like ragged weight tail)
])
def test_linear_f32(M, K, N_):
    X, W = operands(M, K, N_)
    ref = bf16_np(X) @ bf16_np(W).T
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    out = torch.full((M, N_), float("nan"), device="cuda")
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_F32, out, N_, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    got = out.cpu().numpy()
    assert np.isfinite(got).all()
    assert rowwise_rel(got, ref) < 1e-4


def test_linear_bias_gelu_bf16_and_scatter_add():
    M, K, N_ = 70, 1024, 384
    X, W = operands(M, K, N_, seed=1)
    bias = (torch.randn(N_) * 0.1).to(torch.bfloat16)
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    out = torch.zeros(M, N_, dtype=torch.bfloat16, device="cuda")
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_BIAS_GELU_BF16, out, N_, ws, bias=bias.cuda())
    acc = bf16_np(X) @ bf16_np(W).T + bf16_np(bias)
    ref = torch.nn.functional.gelu(torch.from_numpy(acc)).numpy()
    assert rowwise_rel(bf16_np(out), ref) < 1e-2        # one bf16 rounding of the output
    # residual scatter-add into rows of a larger fp32 matrix; untouched rows stay bit-identical
    h0 = torch.randn(200, N_, device="cuda")
    h = h0.clone()
    rows = torch.randperm(200)[:M].to(torch.int32)
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_ADD_F32, h, N_, ws, rows=rows.cuda())
    torch.cuda.synchronize()
    ref_h = h0.cpu().double().numpy()
    ref_h[rows.numpy()] += bf16_np(X) @ bf16_np(W).T
    assert rowwise_rel(h.cpu().numpy(), ref_h) < 1e-4
    other = np.setdiff1d(np.arange(200), rows.numpy())
    assert torch.equal(h[other], h0[other])
    assert N.spd_workspace_status(ws) == 0


def test_linear_split_tiles_are_deterministic():
    # K split across CTAs (32 weight tiles on every SM): partials summed in CTA order
    M, K, N_ = 256, 4096, 4096
    X, W = operands(M, K, N_, seed=2)
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(3):
        out = torch.empty(M, N_, device="cuda")
        N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_F32, out, N_, ws)
        outs.append(out)
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


@pytest.mark.parametrize("M,K,N_,epi", [
    (256, 1024, 22016, N.EPI_F32),      # CTA pairs, stream-K (86 pair tiles > 76 pair slots)
    (300, 1024, 12288, N.EPI_F32),      # stream-K over two token tiles (96 tiles)
    (256, 1024, 40960, N.EPI_F32),      # CTA pairs, stream-K over 160 pair tiles
    (256, 4096, 12288, N.EPI_F32),      # CTA pairs, one tile per pair (48 pair tiles)
    (230, 2048, 11008, N.EPI_F32),      # CTA pairs, stream-K, ragged token tile halves
    (200, 4096, 4096, N.EPI_ADD_F32),   # CTA pairs, split-K with red.add
    (160, 11008, 4096, N.EPI_ADD_F32),  # CTA pairs, split-K, long K
])
@pytest.mark.parametrize("determ", [0, 1])
def test_linear_cta_pairs(M, K, N_, epi, determ):
    X, W = operands(M, K, N_, seed=M + K)
    ref = bf16_np(X) @ bf16_np(W).T
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    h0 = torch.randn(M, N_, device="cuda") if epi == N.EPI_ADD_F32 else torch.zeros(M, N_, device="cuda")
    outs = []
    N.spd_set_deterministic(determ)
    try:
        for _ in range(2):
            out = h0.clone() if epi == N.EPI_ADD_F32 else torch.full((M, N_), float("nan"), device="cuda")
            N.spd_linear(X.cuda(), M, K, W.cuda(), N_, epi, out, N_, ws)
            torch.cuda.synchronize()
            assert N.spd_workspace_status(ws) == 0
            outs.append(out)
    finally:
        N.spd_set_deterministic(0)
    want = ref + (h0.cpu().double().numpy() if epi == N.EPI_ADD_F32 else 0.0)
    for out in outs:
        got = out.cpu().numpy()
        assert np.isfinite(got).all()
        assert rowwise_rel(got, want) < 1e-4
    if determ:  # every element summed in a fixed order: bit-identical runs
        assert torch.equal(outs[0], outs[1])


@pytest.mark.parametrize("M", [1, 2, 3, 4])
@pytest.mark.parametrize("K,N_", [(256, 1000), (4096, 4096), (11008, 640)])
def test_linear_few_tokens_matrix_vector_path(M, K, N_):
    # at most four tokens with K a multiple of 256: the matrix-vector kernel (F32 output, and the
    # residual scatter-add, whose K range is split over several CTAs)
    X, W = operands(M, K, N_, seed=M + K)
    ref = bf16_np(X) @ bf16_np(W).T
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    out = torch.full((M, N_), float("nan"), device="cuda")
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_F32, out, N_, ws)
    h0 = torch.randn(9, N_, device="cuda")
    h = h0.clone()
    rows = torch.randperm(9)[:M].to(torch.int32)
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, N.EPI_ADD_F32, h, N_, ws, rows=rows.cuda())
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    assert rowwise_rel(out.cpu().numpy(), ref) < 1e-4
    ref_h = h0.cpu().double().numpy()
    ref_h[rows.numpy()] += ref
    assert rowwise_rel(h.cpu().numpy(), ref_h) < 1e-4
    other = np.setdiff1d(np.arange(9), rows.numpy())
    assert torch.equal(h[other], h0[other])
