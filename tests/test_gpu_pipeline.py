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
