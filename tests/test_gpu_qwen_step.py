"""The whole SPIDER step at the Qwen2-style GQA shape (dynamic resolution, received-attention form)
against the oracle's stages: 4 requests of 256-1024 post-merger visual tokens of width 1280 (an
encoder without [CLS]: the received-attention form of Sec. 4.1.1), each pruned to a quarter, the
1280 -> 3584 -> 3584 projector, 256 text tokens per request, then 2 decoder layers of width 3584 with
28 query and 4 KV heads of 128, FFN 18944, theta 1e6, eps 1e-6, vocabulary 152064.

Kept indices bit-exact (well-conditioned seeded images); the decoder compared on a plan in which
every token bypasses both sub-layers except, per sequence, sampled visual and text tokens with mixed
attention-only / FFN-only / both targets and the last token (K and V of every token are computed
and used; see test_gpu_prefill._sampled_plan); hidden states and logits within 2e-2 normwise per
row, from the oracle's own projector output; the bypassed rows bit-identical to their inputs."""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N
from paper_2609_34977_gb300 import synth
from paper_2609_34977_gb300.pipeline import VarResSpiderPrefill
from tests.gpu_util import bf16_np, conditioned_vision, rowwise_rel

pytestmark = pytest.mark.gpu
TOL = 2e-2


def test_qwen2_shaped_spider_step():
    cfg = dict(synth.QWEN2_DECODER, n_layers=2)
    w = synth.decoder_weights(20260301, cfg, device="cuda")
    model = N.SpdModel(cfg, w)
    n_patches, n_text = [256, 512, 768, 1024], [256] * 4
    vis_in, kept = [], []
    for b, n in enumerate(n_patches):
        _, v, res = conditioned_vision(20260310 + 100 * b, 1, n, 1280, 2, 16, n // 4, 1, has_cls=False,
                                       attn_form=1)
        vis_in.append(v)
        kept.append(res[0]["keep_idx"])
    pipe = VarResSpiderPrefill(model, n_patches=n_patches, d_vis=1280, n_feat_layers=2, final_layer=1,
                               n_heads_vis=16, keep_ratio=0.25, text_lens=n_text)
    assert pipe.keeps == [n // 4 for n in n_patches]
    lens = [k + t for k, t in zip(pipe.keeps, n_text)]
    r = np.random.default_rng(20260399)
    mask = np.full((2, pipe.T), 3, np.uint8)
    start = 0
    for n, v in zip(lens, pipe.keeps):
        rows = np.r_[r.choice(v, 6, replace=False), v + r.choice(n - v, 6, replace=False)]
        mask[:, start + rows] = r.integers(0, 3, size=(2, len(rows)))
        mask[:, start + n - 1] = 0
        start += n
    text = synth.text_embeddings(20260398, sum(n_text), 3584)
    feats = [[torch.from_numpy(f).cuda() for f in v["feats"]] for v in vis_in]
    attn = [torch.from_numpy(v["attn"]).cuda() for v in vis_in]
    logits = pipe.run(feats, attn, torch.from_numpy(text.view(np.int16)).view(torch.bfloat16).cuda(), mask)
    torch.cuda.synchronize()
    assert pipe.status() == 0
    for b in range(4):
        np.testing.assert_array_equal(pipe.keep_idx[b].cpu().numpy(), kept[b])
    # oracle: kept final-layer rows in bf16, projector, [visual; text] per request, prefill
    om = od.model_from_torch(w, cfg)
    del w
    xv = od.project(om, np.concatenate([od.bf16_round(v["feats"][1][0][k]) for v, k in zip(vis_in, kept)]))
    tx = synth.bf16_bits_to_f32(text).astype(np.float64)
    parts, vo, to = [], 0, 0
    for k, t in zip(pipe.keeps, n_text):
        parts += [xv[vo:vo + k], tx[to:to + t]]
        vo, to = vo + k, to + t
    x = np.concatenate(parts)
    got_x = bf16_np(pipe.x)
    assert np.array_equal(got_x[~pipe.token_is_visual], x[~pipe.token_is_visual])
    assert rowwise_rel(got_x[pipe.token_is_visual], x[pipe.token_is_visual]) < 1e-2
    h_o, lg_o = od.prefill(om, x, pipe.cu, mask)
    h = pipe.h.cpu().numpy()
    assert rowwise_rel(h, h_o) < TOL
    assert rowwise_rel(logits.cpu().numpy(), lg_o) < TOL
    bypass = np.flatnonzero((mask == 3).all(axis=0))
    np.testing.assert_array_equal(h[bypass], got_x[bypass])
