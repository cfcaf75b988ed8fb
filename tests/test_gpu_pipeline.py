"""The whole SPIDER step (Alg. 1: MSV-Prune, gather, projector, sequence assembly, decoder prefill
with the adaptive skip plan, LM head) at the benchmark's shapes, against the oracle's stages in the
same order: the LLaVA-1.5-7B shape (one tile of 1 + 576 patches x 1024 at ViT layers 12 and 24, 16
heads, keep 192 with r = 0.7 and K = 4, projector 1024 -> 4096 -> 4096, 64 text tokens, decoder
layers of width 4096 with 32 heads and FFN 11008, vocabulary 32000), with 2 of the 32 decoder layers
(every layer has the same shapes and launch configuration; the oracle's fp64 weights of all 32 would
take 52 GB of host memory).

Kept indices bit-exact (a well-conditioned seeded tile); projector rows within one bf16 rounding
(1e-2 normwise); hidden states and logits within 2e-2 (normwise per row), end to end from the
oracle's own projector output."""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N
from paper_2609_34977_gb300 import synth
from paper_2609_34977_gb300.pipeline import SpiderPrefill
from tests.gpu_util import bf16_np, conditioned_vision, rowwise_rel

pytestmark = pytest.mark.gpu
TOL = 2e-2


def test_spider_step_at_the_llava15_shape():
    L, keep, n_text = 2, 192, 64
    cfg = dict(synth.LLAVA_7B_DECODER, n_layers=L)
    w = synth.decoder_weights(20260001, cfg, device="cuda")  # std 0.02, as in the benchmark
    wd = {k: v for k, v in w.items() if k != "layers"}
    wd["layers"] = w["layers"]
    model = N.SpdModel(cfg, wd)
    seed, v, res = conditioned_vision(20260101, 1, 576, 1024, 2, 16, keep, 1)
    pipe = SpiderPrefill(model, n_patch=576, has_cls=True, d_vis=1024, n_feat_layers=2, final_layer=1,
                         n_heads_vis=16, attn_form=0, keep=keep, tiles_per_req=[1], text_lens=[n_text])
    m_llava = synth.skip_targets("llava-1.5-7b")[:L]
    admit, target = synth.adaptive_plan(seed, L, pipe.token_is_visual, 0.9, m_llava, 0, L)
    mask = N.spd_plan_adaptive(L, admit, target)
    text = synth.text_embeddings(seed, n_text, 4096)
    feats = [torch.from_numpy(f).cuda() for f in v["feats"]]
    logits = pipe.run(feats, torch.from_numpy(v["attn"]).cuda(),
                      torch.from_numpy(text.view(np.int16)).view(torch.bfloat16).cuda(), mask)
    torch.cuda.synchronize()
    assert pipe.status() == 0
    kept = res[0]["keep_idx"]
    np.testing.assert_array_equal(pipe.keep_idx.cpu().numpy()[0], kept)
    # oracle: the kept final-layer rows in bf16, the projector, [visual; text], the prefill
    om = od.model_from_torch(w, cfg)
    vis = od.bf16_round(v["feats"][1][0, 1 + kept])
    x = np.concatenate([od.project(om, vis), synth.bf16_bits_to_f32(text).astype(np.float64)])
    # the decoder's input rows: the text rows exactly, the projector's within its bf16 roundings
    assert np.array_equal(bf16_np(pipe.x)[keep:], x[keep:])
    assert rowwise_rel(bf16_np(pipe.x)[:keep], x[:keep]) < 1e-2
    h_o, lg_o = od.prefill(om, x, pipe.cu, od.expand_adaptive_plan(admit, target, L))
    assert rowwise_rel(pipe.h.cpu().numpy(), h_o) < TOL
    assert rowwise_rel(logits.cpu().numpy(), lg_o) < TOL


@pytest.mark.parametrize("host", [True, False])
def test_whole_step_entry_with_host_or_device_buffers(host):
    # spd_step (one C-ABI call: prune, gather, projector, text rows, prefill) with the inputs and
    # the logits in pinned host memory (copied inside the call) or on the device, against the
    # oracle's stages on the tiny decoder with a projector: 2 requests of 1 and 2 tiles
    cfg = dict(synth.TINY_DECODER, d_vis=128, d_proj=192)
    w = synth.decoder_weights(20260501, cfg, std=0.05)
    model = N.SpdModel(cfg, {k: (v.cuda() if k != "layers" else [{kk: vv.cuda() for kk, vv in lw.items()}
                                                                  for lw in v]) for k, v in w.items()})
    keep, tiles, texts = 32, [1, 2], [16, 8]
    seed, v, res = conditioned_vision(20260510, 3, 576, 128, 2, 8, keep, 1)
    pc = N.prune_cfg(3, 577, 128, 2, 1, 8, keep)
    text = synth.text_embeddings(seed, sum(texts), 256)
    T = sum(t * keep for t in tiles) + sum(texts)
    vis = np.concatenate([np.r_[np.ones(t * keep, bool), np.zeros(x, bool)] for t, x in zip(tiles, texts)])
    mask = N.spd_plan_static(np.array([1, 2], np.uint8), vis.astype(np.uint8))
    feats = [torch.from_numpy(f) for f in v["feats"]]
    attn = torch.from_numpy(v["attn"])
    tx = torch.from_numpy(text.view(np.int16)).view(torch.bfloat16)
    if host:
        feats, attn, tx = [f.pin_memory() for f in feats], attn.pin_memory(), tx.pin_memory()
        logits = torch.full((2, 512), float("nan")).pin_memory()
    else:
        feats, attn, tx = [f.cuda() for f in feats], attn.cuda(), tx.cuda()
        logits = torch.full((2, 512), float("nan"), device="cuda")
    ws = torch.zeros(N.spd_step_workspace_size(model, pc, tiles, texts), dtype=torch.uint8, device="cuda")
    N.spd_step(model, pc, tiles, texts, feats, attn, tx, mask, logits, ws)
    torch.cuda.synchronize()
    assert N.spd_step_status(ws, model, pc, tiles, texts) == 0
    om = od.model_from_torch(w, cfg)
    xv = od.project(om, np.concatenate([od.bf16_round(v["feats"][1][t, 1 + res[t]["keep_idx"]]) for t in range(3)]))
    txt = synth.bf16_bits_to_f32(text).astype(np.float64)
    x = np.concatenate([xv[:keep], txt[:16], xv[keep:], txt[16:]])
    cu = [0, keep + 16, T]
    _, lg_o = od.prefill(om, x, cu, mask)
    assert rowwise_rel(logits.cpu().numpy(), lg_o) < TOL


def test_whole_step_entry_equals_the_staged_calls_at_llava_width():
    # spd_step with pinned host buffers at the LLaVA-1.5 shape (one tile, keep 192, projector
    # 1024 -> 4096 -> 4096, 64 text tokens, 2 full-width decoder layers with a skip plan) against the
    # same stages called one by one (SpiderPrefill): bit-identical logits in deterministic mode
    L, keep, n_text = 2, 192, 64
    cfg = dict(synth.LLAVA_7B_DECODER, n_layers=L, vocab=4096)
    w = synth.decoder_weights(20261501, cfg, device="cuda")
    model = N.SpdModel(cfg, w)
    seed, v, res = conditioned_vision(20261510, 1, 576, 1024, 2, 16, keep, 1)
    pipe = SpiderPrefill(model, n_patch=576, has_cls=True, d_vis=1024, n_feat_layers=2, final_layer=1,
                         n_heads_vis=16, attn_form=0, keep=keep, tiles_per_req=[1], text_lens=[n_text])
    admit, target = synth.adaptive_plan(seed, L, pipe.token_is_visual, 0.9,
                                        synth.skip_targets("llava-1.5-7b")[:L], 0, L)
    mask = N.spd_plan_adaptive(L, admit, target)
    text = synth.text_embeddings(seed, n_text, 4096)
    tx = torch.from_numpy(text.view(np.int16)).view(torch.bfloat16)
    pc = N.prune_cfg(1, 577, 1024, 2, 1, 16, keep)
    ws = torch.zeros(N.spd_step_workspace_size(model, pc, [1], [n_text]), dtype=torch.uint8, device="cuda")
    feats_h = [torch.from_numpy(f).pin_memory() for f in v["feats"]]
    attn_h = torch.from_numpy(v["attn"]).pin_memory()
    logits_h = torch.full((1, 4096), float("nan")).pin_memory()
    N.spd_set_deterministic(1)
    try:
        ref = pipe.run([f.cuda() for f in feats_h], attn_h.cuda(), tx.cuda(), mask).clone()
        N.spd_step(model, pc, [1], [n_text], feats_h, attn_h, tx.pin_memory(), mask, logits_h, ws)
        torch.cuda.synchronize()
    finally:
        N.spd_set_deterministic(0)
    assert pipe.status() == 0 and N.spd_step_status(ws, model, pc, [1], [n_text]) == 0
    assert torch.equal(logits_h, ref.cpu())
