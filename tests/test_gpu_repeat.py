"""Repeated runs with programmatic overlap of every launch (each kernel may be scheduled while its
predecessors in the stream still run, and orders itself with the grid dependency wait).

The decoder prefill with sub-layer skipping (Sec. 3.2, Alg. 1 stage 2) is run 30 times back to back
on the same inputs, with the plan given, with the online ASL-Skip plan decided on the host, and with
it decided on the device (admissions and row lists written by kernels and read several launches
later). Every repeat is compared with the oracle (2e-2, normwise per row) and with the first repeat
of its kind (two bf16 units of a row's largest entry: the split-K residual adds land in any order).
A stale or early read anywhere in the chain of launches shows up as a row far outside both.

Two shapes: the whole SPIDER step at the LLaVA-1.5 width (prune of a 1 + 576 x 1024 tile keeping
192, projector 1024 -> 4096 -> 4096, 64 text tokens, 2 decoder layers of width 4096), and the small
6-layer decoder whose online plan spans three decision layers (three list blocks built by kernels).
"""
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
SAME_EXECUTOR = 2.0**-6
REPEATS = 30


def _check_repeats(hs, lgs, h_o, lg_o):
    for k, (h, lg) in enumerate(zip(hs, lgs)):
        assert np.isfinite(h).all() and np.isfinite(lg).all(), k
        eh, el = rowwise_rel(h, h_o), rowwise_rel(lg, lg_o)
        assert eh < TOL and el < TOL, (k, eh, el)
        dh, dl = rowwise_rel(h, hs[0]), rowwise_rel(lg, lgs[0])
        assert dh < SAME_EXECUTOR and dl < SAME_EXECUTOR, (k, dh, dl)


def _layer0_threshold(om, x, cu, vis, slc, w1, w2):
    """A T_skip between two layer-0 values of w1 S_sa + w2 SLC^Norm(0) that lie far apart, with
    tokens on both sides (the decision at layer 0 is then well conditioned)."""
    T = len(x)
    seq_of = np.zeros(T, np.int64)
    for b in range(len(cu) - 1):
        seq_of[cu[b]:cu[b + 1]] = b
    text_rows = [np.flatnonzero((seq_of == b) & ~vis) for b in range(len(cu) - 1)]
    cand = np.flatnonzero(vis)
    s_sa, _, _ = od.skippability(om, np.asarray(x, np.float64), cand, seq_of, text_rows)
    s = np.sort(w1 * s_sa + w2 * slc[0])
    lo, hi = len(s) // 5, len(s) - len(s) // 5
    gaps = s[lo + 1:hi] - s[lo:hi - 1]
    j = lo + int(np.argmax(gaps))
    return 0.5 * (s[j] + s[j + 1]), float(gaps.max())


def test_llava_width_spider_step_repeated_with_overlap():
    L, keep, n_text = 2, 192, 64
    cfg = dict(synth.LLAVA_7B_DECODER, n_layers=L, vocab=4096)
    w = synth.decoder_weights(20260011, cfg, device="cuda")
    w["lm_head"] = (w["lm_head"].float() * 12.0).to(torch.bfloat16)  # peaked vocabularies: E_ii varies
    model = N.SpdModel(cfg, w)
    seed, v, res = conditioned_vision(20260201, 1, 576, 1024, 2, 16, keep, 1)
    pipe = SpiderPrefill(model, n_patch=576, has_cls=True, d_vis=1024, n_feat_layers=2, final_layer=1,
                         n_heads_vis=16, attn_form=0, keep=keep, tiles_per_req=[1], text_lens=[n_text])
    m_llava = synth.skip_targets("llava-1.5-7b")[:L]
    admit, target = synth.adaptive_plan(seed, L, pipe.token_is_visual, 0.9, m_llava, 0, L)
    mask = N.spd_plan_adaptive(L, admit, target)
    text = synth.text_embeddings(seed, n_text, 4096)
    feats = [torch.from_numpy(f).cuda() for f in v["feats"]]
    attn = torch.from_numpy(v["attn"]).cuda()
    text_d = torch.from_numpy(text.view(np.int16)).view(torch.bfloat16).cuda()

    om = od.model_from_torch(w, cfg)
    kept = res[0]["keep_idx"]
    xv = od.project(om, od.bf16_round(v["feats"][1][0, 1 + kept]))
    x = np.concatenate([xv, synth.bf16_bits_to_f32(text).astype(np.float64)])
    cu, vis = pipe.cu, pipe.token_is_visual

    # given plan: 30 steps enqueued back to back, each leaving h and the logits in its own slot
    hs, lgs = [], []
    for _ in range(REPEATS):
        pipe.run(feats, attn, text_d, mask)
        hs.append(pipe.h.clone())
        lgs.append(pipe.logits.clone())
    torch.cuda.synchronize()
    assert pipe.status() == 0
    np.testing.assert_array_equal(pipe.keep_idx.cpu().numpy()[0], kept)
    h_o, lg_o = od.prefill(om, x, cu, od.expand_adaptive_plan(admit, target, L))
    _check_repeats([t.cpu().numpy() for t in hs], [t.cpu().numpy() for t in lgs], h_o, lg_o)

    # online plan (window 1), host and device decisions, on the oracle's own decoder input rows
    # (bf16 values, so both sides start from the same x and take the same layer-0 decisions)
    slc = np.array([0.3, 0.6])
    tgt = np.asarray(m_llava, np.uint8)
    t_skip, gap = _layer0_threshold(om, x, cu, vis, slc, 3.0, 1.0)
    # the GPU's S_sa differs from the oracle's by about 1e-4 (fp32 entropy and cosine of the same
    # bf16 operands): a gap of 6e-3 leaves each decision a margin thirty times that
    assert gap > 6e-3, gap
    h_a, lg_a, admit_a, _, margin = od.prefill_adaptive(om, x, cu, vis, slc, tgt, t_skip, 3.0, 1.0, 1)
    assert margin > 3e-3 and (admit_a[vis] == 0).any() and (admit_a[vis] < 0).any()
    T = len(x)
    xd = torch.from_numpy(x).to(torch.bfloat16).cuda()
    ws = torch.zeros(N.spd_prefill_adaptive_workspace_size(model, T, 1), dtype=torch.uint8, device="cuda")
    for device_plan in (0, 1):
        hs, lgs = [], []
        for _ in range(REPEATS):
            h = torch.full((T, 4096), float("nan"), device="cuda")
            logits = torch.full((1, cfg["vocab"]), float("nan"), device="cuda")
            got = N.spd_prefill_adaptive(model, xd, T, cu, vis, slc, tgt, t_skip, 3.0, 1.0, 1, h, logits,
                                         ws, device_plan=device_plan)
            np.testing.assert_array_equal(got.astype(np.int64), admit_a)
            hs.append(h.cpu().numpy())
            lgs.append(logits.cpu().numpy())
        assert N.spd_workspace_status(ws) == 0
        _check_repeats(hs, lgs, h_a, lg_a)


def test_deterministic_mode_gives_bit_identical_prefills():
    # spd_set_deterministic(1): every GEMM sums in a fixed order (partial slots in CTA order, one
    # read-modify-write per residual element): repeated prefills agree bit for bit, and with the
    # oracle as in the default mode. Two LLaVA-width layers with a skip plan on the visual tokens
    # (fused QKV over 256 tokens, pair tiles split over K, the residual GEMMs' split tiles).
    cfg = dict(n_layers=2, d_model=4096, n_heads=32, n_kv_heads=32, head_dim=128, d_ffn=11008,
               vocab=1000, rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
    w = synth.decoder_weights(41, cfg, std=0.02, device="cuda")
    model = N.SpdModel(cfg, w)
    om = od.model_from_torch(w, cfg)
    T = 256
    x = torch.randn(T, 4096, generator=torch.Generator().manual_seed(42)).to(torch.bfloat16)
    r = np.random.default_rng(43)
    mask = np.zeros((2, T), np.uint8)
    mask[:, :192] = r.integers(0, 4, size=(2, 192))
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, 1), dtype=torch.uint8, device="cuda")
    xd = x.cuda()
    outs = []
    N.spd_set_deterministic(1)
    try:
        for _ in range(5):
            h = torch.full((T, 4096), float("nan"), device="cuda")
            lg = torch.full((1, 1000), float("nan"), device="cuda")
            N.spd_prefill(model, xd, T, [0, T], mask, h, lg, ws)
            outs.append((h, lg))
        torch.cuda.synchronize()
        assert N.spd_workspace_status(ws) == 0
    finally:
        N.spd_set_deterministic(0)
    for h, lg in outs[1:]:
        assert torch.equal(h, outs[0][0]) and torch.equal(lg, outs[0][1])
    h0, lg0 = od.prefill(om, bf16_np(x), [0, T], mask)
    assert rowwise_rel(outs[0][0].cpu().numpy(), h0) < TOL
    assert rowwise_rel(outs[0][1].cpu().numpy(), lg0) < TOL
