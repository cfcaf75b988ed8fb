"""Every output of the C ABI written between guard bands: each output buffer is a view into a larger
allocation whose rows (or elements) before and after it, and the padding columns of a row stride
wider than the row, hold canary values that must come back bit-for-bit untouched. The results inside
are checked too: against the plain product (GEMMs), the oracle (attention), or, in deterministic mode
(every sum in a fixed order), bit for bit against the same call on buffers without guards.

Shapes: the GEMM schedules at the LLaVA-1.5 decoder width (one tile per CTA pair, stream-K, tiles +
remainder, split-K residual reductions with 16-byte and scalar adds, the few-token matrix-vector
kernel), the whole step at the LLaVA-1.5 width with 2 decoder layers (prune, gather, projector, text
rows, prefill), the KV-cache prefill and a decode step, the attention step and the received
attention."""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N
from paper_2609_34977_gb300 import synth
from paper_2609_34977_gb300.pipeline import SpiderPrefill
from tests.gpu_util import bf16_np, conditioned_vision, rowwise_rel

pytestmark = pytest.mark.gpu
G = 3  # guard rows before and after every row-structured output


def _guarded(rows, cols, dtype, canary, pad_cols=0):
    """A [G + rows + G][cols + pad_cols] buffer filled with the canary; returns (buffer, view of
    the rows in the middle)."""
    b = torch.full((G + rows + G, cols + pad_cols), canary, dtype=dtype, device="cuda")
    return b, b[G:G + rows]


def _untouched(b, rows, cols, canary):
    c = torch.full((), canary, dtype=b.dtype, device="cuda")
    head, tail = b[:G], b[G + rows:]
    ok = bool((head == c).all()) and bool((tail == c).all())
    if b.shape[1] > cols:
        ok = ok and bool((b[G:G + rows, cols:] == c).all())
    return ok


def _operands(M, K, N_, seed):
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn(M, K, generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N_, K, generator=g) * 0.02).to(torch.bfloat16)
    return X, W


@pytest.mark.parametrize("M,K,N_,epi,pad", [
    (256, 4096, 12288, N.EPI_F32, 8),        # CTA pairs, one tile per pair
    (256, 1024, 22016, N.EPI_F32, 4),        # CTA pairs, tiles + remainder (86 pair tiles)
    (300, 1024, 12288, N.EPI_BF16, 8),       # stream-K over two token tiles, bf16 output
    (200, 4096, 4096, N.EPI_ADD_F32, 4),     # split-K residual, 16-byte reductions
    (200, 4096, 4096, N.EPI_ADD_F32, 3),     # split-K residual, scalar reductions (odd stride)
    (3, 4096, 4096, N.EPI_ADD_F32, 5),       # matrix-vector kernel, residual, split over K
    (2, 256, 1000, N.EPI_F32, 24),           # matrix-vector kernel, F32
])
def test_linear_outputs_between_guard_rows_and_columns(M, K, N_, epi, pad):
    X, W = _operands(M, K, N_, M + K + N_)
    ref = bf16_np(X) @ bf16_np(W).T
    is_bf16 = epi == N.EPI_BF16
    dt = torch.bfloat16 if is_bf16 else torch.float32
    canary = -3.0 if is_bf16 else -12345.0
    b, out = _guarded(M, N_, dt, canary, pad)
    h0 = None
    if epi == N.EPI_ADD_F32:
        h0 = torch.randn(M, N_, device="cuda")
        out[:, :N_] = h0
    ws = torch.zeros(N.spd_linear_workspace_size(M, N_), dtype=torch.uint8, device="cuda")
    N.spd_linear(X.cuda(), M, K, W.cuda(), N_, epi, out, N_ + pad, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    assert _untouched(b, M, N_, canary)
    got = out[:, :N_].float().cpu().numpy().astype(np.float64)
    want = ref + (h0.cpu().double().numpy() if h0 is not None else 0.0)
    assert rowwise_rel(got, want) < (1e-2 if is_bf16 else 1e-4)


def test_whole_step_at_llava_width_between_guard_rows():
    # prune (kept indices, kinds, clusters, scores), gather, projector rows, text rows, the
    # prefill's residual stream and logits: every output between guards; in deterministic mode the
    # guarded run equals an unguarded one bit for bit
    L, keep, n_text = 2, 192, 64
    cfg = dict(synth.LLAVA_7B_DECODER, n_layers=L, vocab=4096)
    w = synth.decoder_weights(20261201, cfg, device="cuda")
    model = N.SpdModel(cfg, w)
    seed, v, res = conditioned_vision(20261210, 1, 576, 1024, 2, 16, keep, 1)
    feats = [torch.from_numpy(f).cuda() for f in v["feats"]]
    attn = torch.from_numpy(v["attn"]).cuda()
    pc = N.prune_cfg(1, 577, 1024, 2, 1, 16, keep)
    text = torch.from_numpy(synth.text_embeddings(seed, n_text, 4096).view(np.int16)).view(torch.bfloat16).cuda()
    pipe = SpiderPrefill(model, n_patch=576, has_cls=True, d_vis=1024, n_feat_layers=2, final_layer=1,
                         n_heads_vis=16, attn_form=0, keep=keep, tiles_per_req=[1], text_lens=[n_text])
    admit, target = synth.adaptive_plan(seed, L, pipe.token_is_visual, 0.9,
                                        synth.skip_targets("llava-1.5-7b")[:L], 0, L)
    mask = N.spd_plan_adaptive(L, admit, target)
    T, D = pipe.T, 4096
    N.spd_set_deterministic(1)
    try:
        ref = pipe.run(feats, attn, text, mask).clone()
        torch.cuda.synchronize()
        assert pipe.status() == 0
        ref_h, ref_x = pipe.h.clone(), pipe.x.clone()
        # the same stages, outputs between guards
        ws_p = torch.zeros(N.spd_prune_workspace_size(pc), dtype=torch.uint8, device="cuda")
        kb, keep_idx = _guarded(1, keep, torch.int32, -7)
        sb, scores = _guarded(1, 576, torch.float32, -1234.5)
        knd_b, kind = _guarded(1, 576, torch.uint8, 9)
        cb, clus = _guarded(1, 576, torch.int8, 99)
        N.spd_prune(pc, feats, attn, keep_idx, kind, clus, scores, ws=ws_p)
        vb, vis = _guarded(keep, 1024, torch.bfloat16, 3.0)
        N.spd_gather_rows_bf16(feats[1], 1, 577, 1024, 1, keep_idx, keep, vis, ws=ws_p)
        xb, x = _guarded(T, D, torch.bfloat16, 5.0)
        ws_j = torch.zeros(N.spd_project_workspace_size(model, keep), dtype=torch.uint8, device="cuda")
        N.spd_project(model, vis, keep, pipe.vis_rows, x, ws_j)
        N.spd_scatter_rows(model, text, n_text, pipe.text_rows, x)
        hb, h = _guarded(T, D, torch.float32, -777.0)
        lb, lg = _guarded(1, 4096, torch.float32, -888.0)
        ws_f = torch.zeros(N.spd_prefill_workspace_size(model, T, 1), dtype=torch.uint8, device="cuda")
        N.spd_prefill(model, x, T, pipe.cu, mask, h, lg, ws_f)
        torch.cuda.synchronize()
        for w_ in (ws_p, ws_j, ws_f):
            assert N.spd_workspace_status(w_) == 0
    finally:
        N.spd_set_deterministic(0)
    assert _untouched(kb, 1, keep, -7) and _untouched(sb, 1, 576, -1234.5)
    assert _untouched(knd_b, 1, 576, 9) and _untouched(cb, 1, 576, 99)
    assert _untouched(vb, keep, 1024, 3.0) and _untouched(xb, T, D, 5.0)
    assert _untouched(hb, T, D, -777.0) and _untouched(lb, 1, 4096, -888.0)
    np.testing.assert_array_equal(keep_idx.cpu().numpy()[0], res[0]["keep_idx"])
    assert torch.equal(x, ref_x) and torch.equal(h, ref_h) and torch.equal(lg, ref)


def test_kv_cache_and_decode_between_guards():
    # the cache block and the decode logits between guards; a decode step's logits against the
    # oracle's prefill of the extended sequences
    cfg = dict(synth.TINY_DECODER, n_layers=2)
    w = synth.decoder_weights(20261301, cfg, std=0.05)
    model = N.SpdModel(cfg, {k: (v.cuda() if k != "layers" else [{kk: vv.cuda() for kk, vv in lw.items()}
                                                                  for lw in v]) for k, v in w.items()})
    om = od.model_from_torch(w, cfg)
    lens, B, max_len, D, V = [30, 45], 2, 64, cfg["d_model"], cfg["vocab"]
    T = sum(lens)
    g = torch.Generator().manual_seed(20261302)
    x = torch.randn(T, D, generator=g).to(torch.bfloat16)
    cu = np.array([0, 30, 75], np.int32)
    n_cache = N.spd_kv_cache_bytes(model, B, max_len) // 2
    GE = 4096  # guard elements around the cache block
    cache_b = torch.full((GE + n_cache + GE,), 7.0, dtype=torch.bfloat16, device="cuda")
    cache_b[GE:GE + n_cache] = 0.0
    cache = cache_b[GE:GE + n_cache]
    hb, h = _guarded(T, D, torch.float32, -1.0)
    lb, lg = _guarded(B, V, torch.float32, -2.0)
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, B), dtype=torch.uint8, device="cuda")
    N.spd_prefill_kv(model, x.cuda(), T, cu, np.zeros((2, T), np.uint8), h, lg, cache, max_len, ws)
    new = torch.randn(B, D, generator=g).to(torch.bfloat16)
    ob, out = _guarded(B, V, torch.float32, -3.0)
    wsd = torch.zeros(N.spd_decode_workspace_size(model, B), dtype=torch.uint8, device="cuda")
    N.spd_decode(model, new.cuda(), np.array(lens), cache, max_len, out, wsd)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0 and N.spd_workspace_status(wsd) == 0
    assert bool((cache_b[:GE] == 7.0).all()) and bool((cache_b[GE + n_cache:] == 7.0).all())
    assert _untouched(hb, T, D, -1.0) and _untouched(lb, B, V, -2.0) and _untouched(ob, B, V, -3.0)
    xe = np.concatenate([bf16_np(x)[:30], bf16_np(new)[:1], bf16_np(x)[30:], bf16_np(new)[1:]])
    _, lo = od.prefill(om, xe, np.array([0, 31, 77]), np.zeros((2, 77), np.uint8))
    assert rowwise_rel(out.cpu().numpy(), lo) < 2e-2


def test_attention_and_received_attention_between_guards():
    # spd_attention's output rows and spd_received_attention's importance vector between guards
    r = np.random.default_rng(20261401)
    lens, H, Hkv, hd = [100, 157], 4, 2, 64
    T = sum(lens)
    q_rows = np.sort(r.choice(T, 120, replace=False))
    pos = np.concatenate([np.arange(n) for n in lens])
    bf = lambda a: torch.from_numpy(a).float().to(torch.bfloat16)
    q = bf(r.standard_normal((len(q_rows), H * hd)))
    kv = bf(r.standard_normal((T, 2 * Hkv * hd)))
    seq = np.searchsorted([100], q_rows, side="right")
    q_cu = np.array([0, int((seq == 0).sum()), len(q_rows)], np.int32)
    q_pos = pos[q_rows].astype(np.int32)
    cu = np.array([0, 100, T], np.int32)
    ob, o = _guarded(len(q_rows), H * hd, torch.bfloat16, 11.0)
    ws = torch.zeros(N.spd_attention_workspace_size(len(q_rows), 2), dtype=torch.uint8, device="cuda")
    N.spd_attention(q.cuda(), torch.from_numpy(q_pos).cuda(), q_cu, kv.cuda(), cu, H, Hkv, hd, o, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    assert _untouched(ob, len(q_rows), H * hd, 11.0)
    qn, kvn = bf16_np(q), bf16_np(kv)
    want = np.zeros_like(qn)
    for b in range(2):
        a0, a1, t0, t1 = q_cu[b], q_cu[b + 1], cu[b], cu[b + 1]
        want[a0:a1] = od.causal_attention(qn[a0:a1], kvn[t0:t1, :Hkv * hd], kvn[t0:t1, Hkv * hd:],
                                          q_pos[a0:a1], np.arange(t1 - t0), H, Hkv, hd)
    assert rowwise_rel(bf16_np(o), want) < 2e-2
    # received attention: 2 maps of 512 x 512, no merger
    maps = torch.from_numpy(r.random((2, 512, 512)).astype(np.float32)).cuda()
    rb, rout = _guarded(1, 2 * 512, torch.float32, -5.0)
    wsr = torch.zeros(N.spd_received_attention_workspace_size(2, 512, 512), dtype=torch.uint8, device="cuda")
    N.spd_received_attention(maps, rout.view(2, 512), wsr)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(wsr) == 0
    assert _untouched(rb, 1, 2 * 512, -5.0)
    np.testing.assert_allclose(rout.view(2, 512).cpu().numpy(), maps.mean(dim=1).cpu().numpy(), rtol=1e-5)
