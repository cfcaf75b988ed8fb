"""Decoder prefill with sub-layer skipping on the GPU (spd_prefill, spd_project) against the CPU
oracle (Sec. 3.2 VSkip-Attn / VSkip-FFN, Alg. 1 stage 2).

Tolerance (bf16 weights and activations, fp32 accumulation): hidden states and logits within 2e-2,
measured normwise per row, max_j |gpu - oracle| / max_j |oracle|. Rows whose every sub-layer is
skipped must come back bit-identical to the input (the fp32 residual is never touched)."""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N
from paper_2609_34977_gb300 import synth
from tests.gpu_util import bf16_np, rowwise_rel

pytestmark = pytest.mark.gpu
TOL = 2e-2
# Two runs of the same executor on the same plan: the split-K residual adds (red.add) land in any
# order, so the fp32 sums differ in the last bits, and where such a sum sits at a bf16 rounding
# boundary the rounded activation moves by one bf16 unit (2^-8 relative), which moves an output
# row by at most about 2^-7 of its largest entry. Two units bound it; one wrong plan bit moves some
# row by far more (each test checks that with the oracle).
SAME_EXECUTOR = 2.0**-6


def wrong_bit_moves(om, xn, cu, mask, h_ref, rng):
    """The smallest row-relative move of the oracle's output under one flipped plan bit (5 tries)."""
    moves = []
    for _ in range(5):
        m2 = mask.copy()
        m2[rng.integers(0, m2.shape[0]), rng.integers(0, m2.shape[1])] ^= 1 << rng.integers(0, 2)
        moves.append(rowwise_rel(od.prefill(om, xn, cu, m2)[0], h_ref))
    return min(moves)


def build(cfg, seed, std=0.05, device="cpu"):
    w = synth.decoder_weights(seed, cfg, std=std, device=device)
    wd = {k: v for k, v in w.items() if k != "layers"}
    wd = {k: v.cuda() for k, v in wd.items()}
    wd["layers"] = [{k: v.cuda() for k, v in lw.items()} for lw in w["layers"]]
    return N.SpdModel(cfg, wd), od.model_from_torch(w, cfg)


def run(model, x, cu, mask):
    T = x.shape[0]
    B = len(cu) - 1
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, B), dtype=torch.uint8, device="cuda")
    h = torch.full((T, model.cfg["d_model"]), float("nan"), device="cuda")
    logits = torch.full((B, model.cfg["vocab"]), float("nan"), device="cuda")
    N.spd_prefill(model, x, T, cu, mask, h, logits, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    return h.cpu().numpy(), logits.cpu().numpy()


def inputs(T, D, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randn(T, D, generator=g).to(torch.bfloat16)


def check(model, om, x, cu, mask):
    h, lg = run(model, x.cuda(), cu, mask)
    ho, lo = od.prefill(om, bf16_np(x), cu, mask if mask is not None else
                        np.zeros((om["cfg"]["n_layers"], x.shape[0]), np.uint8))
    assert np.isfinite(h).all() and np.isfinite(lg).all()
    eh, el = rowwise_rel(h, ho), rowwise_rel(lg, lo)
    assert eh < TOL and el < TOL, (eh, el)
    return h, lg


def test_tiny_config_static_plan():
    # 2-layer decoder, 64 visual + 32 text tokens, plan {L0: none, L1: skip FFN} on visual tokens.
    model, om = build(synth.TINY_DECODER, 1)
    x = inputs(96, 256, 2)
    vis = np.r_[np.ones(64), np.zeros(32)].astype(np.uint8)
    mask = N.spd_plan_static(np.array([0, 2], np.uint8), vis)
    h, _ = check(model, om, x, [0, 96], mask)


def test_tiny_no_skipping_and_null_mask():
    model, om = build(synth.TINY_DECODER, 3)
    x = inputs(96, 256, 4)
    h1, l1 = check(model, om, x, [0, 96], None)
    h2, l2 = run(model, x.cuda(), [0, 96], np.zeros((2, 96), np.uint8))
    # the same computation, up to the order of the residual adds (SAME_EXECUTOR)
    assert rowwise_rel(h2, h1) < SAME_EXECUTOR and rowwise_rel(l2, l1) < SAME_EXECUTOR


@pytest.mark.parametrize("seed", [5, 6])
def test_adaptive_plan_mixed_targets(seed):
    cfg = dict(synth.TINY_DECODER, n_layers=4)
    model, om = build(cfg, seed)
    T = 150
    x = inputs(T, 256, seed + 10)
    vis = np.r_[np.ones(110, bool), np.zeros(40, bool)]
    admit, target = synth.adaptive_plan(seed, 4, vis, 0.6, np.array([1, 2, 1, 2], np.uint8), 0, 3)
    mask = N.spd_plan_adaptive(4, admit, target)
    assert (mask & 1).any() and (mask & 2).any()
    check(model, om, x, [0, T], mask)


def test_packed_ragged_sequences_and_bypass_is_bit_exact():
    cfg = dict(synth.TINY_DECODER, n_layers=3)
    model, om = build(cfg, 7)
    cu = [0, 70, 71, 200, 333]          # a 1-token sequence, tiles of 64 with ragged tails
    T = cu[-1]
    x = inputs(T, 256, 8)
    r = np.random.default_rng(9)
    mask = r.integers(0, 4, size=(3, T)).astype(np.uint8)
    mask[:, [5, 100, 250]] = 3           # these rows skip every sub-layer of every layer
    mask[:, [69, 70, 199, 332]] = 0      # last tokens of each sequence stay fully active
    h, _ = check(model, om, x, cu, mask)
    for row in (5, 100, 250):
        np.testing.assert_array_equal(h[row], bf16_np(x[row]).astype(np.float32))


def test_gqa_head_dim_128_long_sequence():
    cfg = dict(n_layers=2, d_model=512, n_heads=8, n_kv_heads=2, head_dim=128, d_ffn=1024,
               vocab=1000, rope_theta=1e6, rms_eps=1e-6, d_vis=0, d_proj=0)
    model, om = build(cfg, 11, std=0.03)
    T = 330
    x = inputs(T, 512, 12)
    vis = np.r_[np.ones(250, bool), np.zeros(80, bool)]
    admit, target = synth.adaptive_plan(13, 2, vis, 0.5, np.array([1, 2], np.uint8), 0, 1)
    check(model, om, x, [0, T], N.spd_plan_adaptive(2, admit, target))


def test_skip_attn_row_is_still_a_key_and_value():
    cfg = dict(synth.TINY_DECODER, n_layers=1)
    model, om = build(cfg, 14)
    T, j = 40, 10
    x = inputs(T, 256, 15)
    mask = np.zeros((1, T), np.uint8)
    mask[0, j] = 1
    h1, _ = check(model, om, x, [0, T], mask)
    x2 = x.clone()
    x2[j] = (x2[j].float() + torch.randn(256, generator=torch.Generator().manual_seed(16))).to(torch.bfloat16)
    h2, _ = check(model, om, x2, [0, T], mask)           # the oracle's attention is causal
    assert rowwise_rel(h1[:j], h2[:j]) < SAME_EXECUTOR   # earlier tokens do not see j
    assert np.abs(h1[j + 1:] - h2[j + 1:]).max() > 1e-3  # later tokens read j's K/V


def test_projector():
    cfg = dict(synth.TINY_DECODER, d_vis=128, d_proj=384)
    model, om = build(cfg, 16)
    R = 70
    vis = torch.randn(R, 128).to(torch.bfloat16)
    rows = torch.arange(R, dtype=torch.int32) * 2 + 1
    x = torch.zeros(2 * R + 1, 256, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(N.spd_project_workspace_size(model, R), dtype=torch.uint8, device="cuda")
    N.spd_project(model, vis.cuda(), R, rows.cuda(), x, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    ref = od.project(om, bf16_np(vis))
    got = bf16_np(x)
    assert rowwise_rel(got[rows.numpy()], ref) < TOL
    assert not got[0::2].any()


def test_llava_width_layer_with_cta_pairs():
    # one decoder layer at the LLaVA-1.5-7B width (the benchmark's GEMM shapes: fused QKV over
    # 256 tokens, gate-up, down, O on query/FFN rows), a skip plan on the visual tokens
    cfg = dict(n_layers=1, d_model=4096, n_heads=32, n_kv_heads=32, head_dim=128, d_ffn=11008,
               vocab=1000, rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
    model, om = build(cfg, 21, std=0.02)
    T = 256
    x = inputs(T, 4096, 22)
    vis = np.r_[np.ones(192, bool), np.zeros(64, bool)]
    r = np.random.default_rng(23)
    mask = np.zeros((1, T), np.uint8)
    mask[0, vis] = r.integers(0, 3, size=192)  # some tokens skip attention, some the FFN
    check(model, om, x, [0, T], mask)


def _sampled_plan(lens, n_vis, seed, per_seq=6):
    """Every token bypasses both sub-layers except, per sequence, a few visual and text tokens that
    run attention, the FFN or both (the oracle then computes K and V for every token but queries,
    attention and FFN only for the sampled rows, which keeps a full-width layer cheap on the CPU);
    the last token of each sequence runs both (its logits)."""
    r = np.random.default_rng(seed)
    T = sum(lens)
    mask = np.full((1, T), 3, np.uint8)
    start = 0
    for n, v in zip(lens, n_vis):
        rows = np.r_[r.choice(v, per_seq, replace=False), v + r.choice(n - v, per_seq, replace=False)]
        mask[0, start + rows] = r.integers(0, 3, size=len(rows))
        mask[0, start + n - 1] = 0
        start += n
    return mask


@pytest.mark.parametrize("shape", ["llava-next-7b", "qwen2-gqa"])
def test_full_width_layer_at_serving_token_counts(shape):
    # one decoder layer at the full width of the workload with its token counts: LLaVA-NeXT-7B
    # (8 requests of 320 kept visual + 128 text tokens) and the Qwen2-style GQA decoder (4 requests
    # of 256-1024 kept visual + 256 text tokens, 28 query / 4 KV heads); K and V of all ~3600
    # tokens, sampled query and FFN rows (see _sampled_plan), every row and the logits compared
    if shape == "llava-next-7b":
        cfg = dict(n_layers=1, d_model=4096, n_heads=32, n_kv_heads=32, head_dim=128, d_ffn=11008,
                   vocab=1000, rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
        n_vis, n_text = [320] * 8, [128] * 8
    else:
        cfg = dict(n_layers=1, d_model=3584, n_heads=28, n_kv_heads=4, head_dim=128, d_ffn=18944,
                   vocab=1000, rope_theta=1e6, rms_eps=1e-6, d_vis=0, d_proj=0)
        n_vis, n_text = [256, 512, 768, 1024], [256] * 4
    lens = [v + t for v, t in zip(n_vis, n_text)]
    model, om = build(cfg, 31, std=0.02, device="cuda")  # weights drawn on the GPU (fast)
    T = sum(lens)
    x = inputs(T, cfg["d_model"], 32)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    mask = _sampled_plan(lens, n_vis, 33)
    h, _ = check(model, om, x, cu, mask)
    bypass = np.flatnonzero(mask[0] == 3)
    np.testing.assert_array_equal(h[bypass], bf16_np(x)[bypass])  # the residual passes unchanged


# ---- ASL-Skip online plan (Sec. 4.2, Eq. 6, Alg. 1 stage 2) ----------------------------------------
def _adaptive_inputs(seed, lens, n_text):
    cfg = dict(synth.TINY_DECODER, n_layers=6)
    w = synth.decoder_weights(seed, cfg, std=0.05)
    w["lm_head"] = (w["lm_head"].float() * 12.0).to(torch.bfloat16)  # peaked vocabularies: E_ii varies
    om = od.model_from_torch(w, cfg)
    wd = {k: v.cuda() for k, v in w.items() if k != "layers"}
    wd["layers"] = [{k: v.cuda() for k, v in lw.items()} for lw in w["layers"]]
    model = N.SpdModel(cfg, wd)
    T = sum(lens)
    x = inputs(T, cfg["d_model"], seed + 1)
    vis = np.concatenate([np.r_[np.ones(n - t, bool), np.zeros(t, bool)] for n, t in zip(lens, n_text)])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    return model, om, x, vis, cu


@pytest.mark.parametrize("device_plan", [0, 1])
def test_adaptive_plan_matches_oracle(device_plan):
    model, om, x, vis, cu = _adaptive_inputs(31, [64, 40], [16, 8])
    slc = np.array([0.2, 0.5, 0.1, 0.7, 0.3, 0.9])
    tgt = np.array([1, 2, 1, 1, 2, 2], np.uint8)
    xn = bf16_np(x)
    chosen = None
    for t_skip in np.linspace(0.6, 2.6, 41):  # a threshold every decision clears by a margin
        h0, lg0, admit0, target0, margin = od.prefill_adaptive(om, xn, cu, vis, slc, tgt, t_skip,
                                                               3.0, 1.0, 3)
        if margin > 0.05 and len(set(admit0[vis])) >= 2:
            chosen = (t_skip, h0, lg0, admit0)
            break
    assert chosen is not None, "no well-separated threshold in the grid"
    t_skip, h0, lg0, admit0 = chosen
    T = x.shape[0]
    ws = torch.zeros(N.spd_prefill_adaptive_workspace_size(model, T, len(cu) - 1), dtype=torch.uint8,
                     device="cuda")
    h = torch.full((T, 256), float("nan"), device="cuda")
    logits = torch.full((len(cu) - 1, 512), float("nan"), device="cuda")
    admit = N.spd_prefill_adaptive(model, x.cuda(), T, cu, vis, slc, tgt, t_skip, 3.0, 1.0, 3, h,
                                   logits, ws, device_plan=device_plan)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    np.testing.assert_array_equal(admit.astype(np.int64), admit0)
    assert np.all(admit[~vis] == -1) and np.all(admit < 3)
    assert rowwise_rel(h.cpu().numpy(), h0) < TOL
    assert rowwise_rel(logits.cpu().numpy(), lg0) < TOL


@pytest.mark.parametrize("bits,w1", [
    (N.SPD_SKIP_NO_ENTROPY, 3.0), (N.SPD_SKIP_NO_ITC, 3.0), (N.SPD_SKIP_NO_ACCUM, 3.0),
    (N.SPD_SKIP_NO_SLC, 3.0), (0, 0.0), (N.SPD_SKIP_NO_ACCUM | N.SPD_SKIP_NO_SLC, 3.0)],
    ids=["no_entropy", "no_itc", "no_accum", "no_slc", "no_s_sa", "no_accum_no_slc"])
@pytest.mark.parametrize("device_plan", [0, 1])
def test_adaptive_plan_ablations_match_oracle(bits, w1, device_plan):
    # the ablation variants of the ASL-Skip table against the oracle's, on a threshold that every
    # decision clears by a margin
    model, om, x, vis, cu = _adaptive_inputs(35, [64, 40], [16, 8])
    slc = np.array([0.2, 0.5, 0.1, 0.7, 0.3, 0.9])
    tgt = np.array([1, 2, 1, 1, 2, 2], np.uint8)
    kw = dict(use_entropy=not bits & N.SPD_SKIP_NO_ENTROPY, use_itc=not bits & N.SPD_SKIP_NO_ITC,
              accumulate=not bits & N.SPD_SKIP_NO_ACCUM, use_slc=not bits & N.SPD_SKIP_NO_SLC)
    xn = bf16_np(x)
    chosen = None
    for t_skip in np.linspace(0.15, 6.0, 235):
        h0, lg0, admit0, target0, margin = od.prefill_adaptive(om, xn, cu, vis, slc, tgt, t_skip, w1,
                                                               1.0, 3, **kw)
        varied = len(set(admit0[vis])) >= 2 or (w1 == 0.0 and (admit0 >= 0).any())
        if margin > 0.02 and varied:
            chosen = (t_skip, h0, lg0, admit0, target0)
            break
    assert chosen is not None, "no well-separated threshold in the grid"
    t_skip, h0, lg0, admit0, target0 = chosen
    T = x.shape[0]
    ws = torch.zeros(N.spd_prefill_adaptive_workspace_size(model, T, len(cu) - 1), dtype=torch.uint8,
                     device="cuda")
    h = torch.full((T, 256), float("nan"), device="cuda")
    logits = torch.full((len(cu) - 1, 512), float("nan"), device="cuda")
    admit = N.spd_prefill_adaptive(model, x.cuda(), T, cu, vis, slc, tgt, t_skip, w1, 1.0, 3, h,
                                   logits, ws, ablate=bits, device_plan=device_plan)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    np.testing.assert_array_equal(admit.astype(np.int64), admit0)
    assert rowwise_rel(h.cpu().numpy(), h0) < TOL
    assert rowwise_rel(logits.cpu().numpy(), lg0) < TOL


@pytest.mark.parametrize("seed,lens,n_text", [
    (37, [4, 30], [1, 0]),  # a sequence of visual tokens only (no text mean: F_itc = 1/2)
    (41, [4], [1]),         # four tokens: the matrix-vector path, whose fused norms meet padded lists
])
def test_adaptive_device_plan_small_and_textless_sequences(seed, lens, n_text):
    model, om, x, vis, cu = _adaptive_inputs(seed, lens, n_text)
    slc = np.array([0.2, 0.5, 0.1, 0.7, 0.3, 0.9])
    tgt = np.array([1, 2, 1, 1, 2, 2], np.uint8)
    xn = bf16_np(x)
    chosen = None
    for t_skip in np.linspace(0.15, 6.0, 235):
        h0, lg0, admit0, _, margin = od.prefill_adaptive(om, xn, cu, vis, slc, tgt, t_skip, 3.0, 1.0, 3)
        if margin > 0.02 and (admit0 >= 0).any() and (admit0[vis] < 0).any():
            chosen = (t_skip, h0, lg0, admit0)
            break
    assert chosen is not None, "no well-separated threshold in the grid"
    t_skip, h0, lg0, admit0 = chosen
    T = x.shape[0]
    B = len(lens)
    ws = torch.zeros(N.spd_prefill_adaptive_workspace_size(model, T, B), dtype=torch.uint8, device="cuda")
    h = torch.full((T, 256), float("nan"), device="cuda")
    logits = torch.full((B, 512), float("nan"), device="cuda")
    admit = N.spd_prefill_adaptive(model, x.cuda(), T, cu, vis, slc, tgt, t_skip, 3.0, 1.0, 3, h, logits,
                                   ws, device_plan=1)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    np.testing.assert_array_equal(admit.astype(np.int64), admit0)
    assert rowwise_rel(h.cpu().numpy(), h0) < TOL
    assert rowwise_rel(logits.cpu().numpy(), lg0) < TOL


def test_adaptive_plan_with_given_plan_is_the_plain_prefill():
    # the same tokens, the plan the online rule chose, run through spd_prefill: the same result up
    # to the order of the residual adds (split-K red.add) and the bf16 roundings that order decides
    model, om, x, vis, cu = _adaptive_inputs(33, [48], [16])
    slc = np.full(6, 0.4)
    tgt = np.array([2, 1, 2, 1, 2, 1], np.uint8)
    T = x.shape[0]
    ws = torch.zeros(N.spd_prefill_adaptive_workspace_size(model, T, 1), dtype=torch.uint8, device="cuda")
    h1 = torch.zeros((T, 256), device="cuda")
    lg1 = torch.zeros((1, 512), device="cuda")
    admit = N.spd_prefill_adaptive(model, x.cuda(), T, cu, vis, slc, tgt, 0.9, 3.0, 1.0, 3, h1, lg1, ws)
    torch.cuda.synchronize()
    target = np.where(admit >= 0, tgt[np.maximum(admit, 0)], 0).astype(np.uint8)
    plan = od.expand_adaptive_plan(admit.astype(np.int64), target, 6)
    h2, lg2 = run(model, x.cuda(), cu, plan)
    assert (admit >= 0).any()
    assert rowwise_rel(h1.cpu().numpy(), h2) < SAME_EXECUTOR
    assert rowwise_rel(lg1.cpu().numpy(), lg2) < SAME_EXECUTOR
    h0, _ = od.prefill(om, bf16_np(x), cu, plan)
    assert wrong_bit_moves(om, bf16_np(x), cu, plan, h0, np.random.default_rng(34)) > 3 * SAME_EXECUTOR


# ---- KV cache and decode steps ---------------------------------------------------------------------
def _decode_case(seed, lens, n_vis, n_layers=3, d_ffn=None, **over):
    cfg = dict(synth.TINY_DECODER, n_layers=n_layers, **over)
    if d_ffn:
        cfg["d_ffn"] = d_ffn
    model, om = build(cfg, seed)
    T = sum(lens)
    x = inputs(T, cfg["d_model"], seed + 1)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    vis = np.concatenate([np.r_[np.ones(v, bool), np.zeros(n - v, bool)] for n, v in zip(lens, n_vis)])
    r = np.random.default_rng(seed)
    mask = np.zeros((n_layers, T), np.uint8)
    mask[:, vis] = r.integers(0, 3, size=(n_layers, int(vis.sum())))
    return cfg, model, om, x, cu, mask


def test_prefill_kv_equals_prefill_and_fills_the_cache():
    cfg, model, om, x, cu, mask = _decode_case(41, [30, 45], [20, 30])
    T, B, max_len = x.shape[0], 2, 64
    h0, lg0 = run(model, x.cuda(), cu, mask)
    cache = torch.zeros(N.spd_kv_cache_bytes(model, B, max_len) // 2, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, B), dtype=torch.uint8, device="cuda")
    h = torch.zeros((T, cfg["d_model"]), device="cuda")
    lg = torch.zeros((B, cfg["vocab"]), device="cuda")
    N.spd_prefill_kv(model, x.cuda(), T, cu, mask, h, lg, cache, max_len, ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    # the cache layout moves each sequence's keys to its own slot, which changes how the attention
    # groups keys into blocks (and so where P is rounded to bf16): equal within the tolerance
    assert rowwise_rel(h.cpu().numpy(), h0) < TOL and rowwise_rel(lg.cpu().numpy(), lg0) < TOL
    ho, lo = od.prefill(om, bf16_np(x), cu, mask)
    assert rowwise_rel(h.cpu().numpy(), ho) < TOL and rowwise_rel(lg.cpu().numpy(), lo) < TOL
    kvd = 2 * cfg["n_kv_heads"] * cfg["head_dim"]
    c = bf16_np(cache).reshape(cfg["n_layers"], B, max_len, kvd)
    for b, n in enumerate([30, 45]):
        assert np.abs(c[:, b, :n]).max() > 0 and not c[:, b, n:].any()  # written rows only


@pytest.mark.parametrize("steps,B,d_ffn,over", [
    (1, 2, None, {}), (2, 2, None, {}),  # d_ffn 688: the down projection on the tiled kernel
    (2, 1, 768, {}),                     # every contraction on the one-token matrix-vector kernel
    (1, 3, 768, {}),                     # the few-token matrix-vector kernel (three tokens of four)
    (1, 5, 768, {}),                     # five tokens: the tiled tcgen05 kernel
    (2, 2, 768, dict(n_heads=2, n_kv_heads=1, head_dim=128)),  # head_dim 128, grouped KV heads
])
def test_decode_steps_equal_prefill_of_the_extended_sequences(steps, B, d_ffn, over):
    lens, n_vis = [30, 45, 20, 33, 12][:B], [20, 30, 10, 25, 5][:B]
    cfg, model, om, x, cu, mask = _decode_case(43, lens, n_vis, d_ffn=d_ffn, **over)
    T, max_len, D = x.shape[0], 64, cfg["d_model"]
    cache = torch.zeros(N.spd_kv_cache_bytes(model, B, max_len) // 2, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, B), dtype=torch.uint8, device="cuda")
    h = torch.zeros((T, D), device="cuda")
    lg = torch.zeros((B, cfg["vocab"]), device="cuda")
    N.spd_prefill_kv(model, x.cuda(), T, cu, mask, h, lg, cache, max_len, ws)
    new = inputs(B * steps, D, 44).reshape(steps, B, D)  # generated-token embeddings
    wsd = torch.zeros(N.spd_decode_workspace_size(model, B), dtype=torch.uint8, device="cuda")
    out = torch.full((B, cfg["vocab"]), float("nan"), device="cuda")
    for s in range(steps):
        N.spd_decode(model, new[s].contiguous().cuda(), np.array(lens) + s, cache, max_len, out, wsd)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(wsd) == 0
    # oracle: each sequence extended by its generated tokens (text tokens: no skipping)
    xs, masks, cu_e = [], [], [0]
    for b in range(B):
        xb = bf16_np(x[cu[b]:cu[b + 1]])
        xs.append(np.concatenate([xb] + [bf16_np(new[s, b:b + 1]) for s in range(steps)]))
        masks.append(np.concatenate([mask[:, cu[b]:cu[b + 1]], np.zeros((cfg["n_layers"], steps), np.uint8)], 1))
        cu_e.append(cu_e[-1] + lens[b] + steps)
    _, lo = od.prefill(om, np.concatenate(xs), cu_e, np.concatenate(masks, 1))
    got = out.cpu().numpy()
    assert np.isfinite(got).all()
    assert rowwise_rel(got, lo) < TOL


def test_prefill_admit_form_equals_the_expanded_plan():
    # the contract's per-token plan form (admission layer, frozen target, 3 = both sub-layers)
    model, om, x, vis, cu = _adaptive_inputs(39, [48, 20], [16, 4])
    T = x.shape[0]
    r = np.random.default_rng(40)
    admit = np.where(vis & (r.random(T) < 0.7), r.integers(0, 6, T), -1).astype(np.int16)
    target = r.integers(1, 4, T).astype(np.uint8)
    ws = torch.zeros(N.spd_prefill_workspace_size(model, T, 2), dtype=torch.uint8, device="cuda")
    h = torch.full((T, 256), float("nan"), device="cuda")
    lg = torch.full((2, 512), float("nan"), device="cuda")
    N.spd_prefill_admit(model, x.cuda(), T, cu, admit, target, h, lg, ws)
    assert N.spd_check(ws) == 0
    mask = od.expand_adaptive_plan(admit, target, 6)
    h0, lg0 = od.prefill(om, bf16_np(x), cu, mask)
    assert rowwise_rel(h.cpu().numpy(), h0) < TOL and rowwise_rel(lg.cpu().numpy(), lg0) < TOL
    h2, lg2 = run(model, x.cuda(), cu, mask)
    assert rowwise_rel(h.cpu().numpy(), h2) < SAME_EXECUTOR
    assert wrong_bit_moves(om, bf16_np(x), cu, mask, h0, r) > 3 * SAME_EXECUTOR
