"""Pins of the decoder-prefill oracle (§3.2 VSkip layers, Alg. 1 stage 2) and of the FLOP model.

Expected values come from libraries (torch's bf16 cast and GELU), closed forms (rotation
invariance, one-key attention), an independent textbook forward, and the paper's Table 1 totals.
"""
import numpy as np
import pytest
import torch

from oracle import decoder as od
from paper_2609_34977_gb300 import flops, synth


def tiny_model(seed=5, cfg=None, std=0.05):
    cfg = dict(cfg or synth.TINY_DECODER)
    w = synth.decoder_weights(seed, cfg, std=std)
    return od.model_from_torch(w, cfg), cfg


def test_bf16_round_matches_torch_cast():
    r = np.random.default_rng(0)
    x = np.concatenate([r.standard_normal(20000) * 10.0 ** r.integers(-5, 5, 20000),
                        [0.0, -0.0, 1.0, 1.00390625, 1.01171875]]).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(od.bf16_round(x.astype(np.float64)), ref.astype(np.float64))


def test_rmsnorm_output_has_unit_rms_times_gain():
    r = np.random.default_rng(1)
    h = r.standard_normal((5, 64)) * 3
    g = r.uniform(0.5, 2, 64)
    y = od.rmsnorm(h, g, 0.0)
    np.testing.assert_allclose(np.sqrt(((y / g) ** 2).mean(1)), 1.0, rtol=1e-12)


def test_rope_is_a_rotation_depending_on_relative_position():
    r = np.random.default_rng(2)
    H, hd = 2, 16
    q, k = r.standard_normal((1, H * hd)), r.standard_normal((1, H * hd))
    np.testing.assert_allclose(od.rope(q, np.array([0]), H, hd, 1e4), q, atol=1e-15)
    for p in (1, 7, 300):
        rq = od.rope(q, np.array([p]), H, hd, 1e4)
        np.testing.assert_allclose(np.linalg.norm(rq), np.linalg.norm(q), rtol=1e-12)
    dots = []
    for shift in (0, 5, 123):
        rq = od.rope(q, np.array([9 + shift]), H, hd, 1e4).reshape(H, hd)
        rk = od.rope(k, np.array([4 + shift]), H, hd, 1e4).reshape(H, hd)
        dots.append((rq * rk).sum(1))
    np.testing.assert_allclose(dots[0], dots[1], rtol=1e-10)
    np.testing.assert_allclose(dots[0], dots[2], rtol=1e-10)


def test_rope_pairs_first_and_second_half():
    # rotate-half: dimension j is paired with j + hd/2 (not with j+1); angle pos * theta^(-2j/hd)
    hd = 8
    x = np.zeros((1, hd))
    x[0, 1] = 1.0
    y = od.rope(x, np.array([3]), 1, hd, 100.0)[0]
    ang = 3 * 100.0 ** (-2.0 / hd)
    expect = np.zeros(hd)
    expect[1], expect[5] = np.cos(ang), np.sin(ang)
    np.testing.assert_allclose(y, expect, atol=1e-15)


def test_attention_closed_forms():
    r = np.random.default_rng(3)
    H, hd = 2, 4
    q = r.standard_normal((3, H * hd))
    k = np.tile(r.standard_normal((1, H * hd)), (3, 1))   # identical keys: uniform weights
    v = r.standard_normal((3, H * hd))
    out = od.causal_attention(q, k, v, np.arange(3), np.arange(3), H, H, hd)
    np.testing.assert_allclose(out[0], v[0], atol=1e-15)            # first token sees only itself
    np.testing.assert_allclose(out[2], v.mean(0), atol=1e-14)       # uniform over three keys
    np.testing.assert_allclose(out[1], v[:2].mean(0), atol=1e-14)


def test_gqa_head_grouping():
    r = np.random.default_rng(4)
    H, Hkv, hd = 4, 2, 4
    q = r.standard_normal((2, H * hd))
    k, v = r.standard_normal((2, Hkv * hd)), r.standard_normal((2, Hkv * hd))
    out = od.causal_attention(q, k, v, np.arange(2), np.arange(2), H, Hkv, hd)
    # heads 0,1 read kv head 0; heads 2,3 read kv head 1; first token sees only its own value
    np.testing.assert_allclose(out[0, 0:hd], v[0, 0:hd])
    np.testing.assert_allclose(out[0, hd:2 * hd], v[0, 0:hd])
    np.testing.assert_allclose(out[0, 2 * hd:3 * hd], v[0, hd:2 * hd])


def test_gelu_matches_torch():
    x = np.linspace(-6, 6, 101)
    ref = torch.nn.functional.gelu(torch.from_numpy(x)).numpy()
    np.testing.assert_allclose(od.gelu(x), ref, rtol=1e-12, atol=1e-15)


@pytest.mark.parametrize("kv", [4, 2])
def test_prefill_with_empty_plan_equals_textbook_forward(kv):
    cfg = dict(synth.TINY_DECODER, n_layers=2, d_model=64, n_heads=4, n_kv_heads=kv, head_dim=16,
               d_ffn=96, vocab=50)
    m, cfg = tiny_model(6, cfg)
    T = 9
    x = od.bf16_round(np.random.default_rng(7).standard_normal((T, 64)))
    mask = np.zeros((2, T), dtype=np.uint8)
    for rnd in (od.identity, od.bf16_round):
        h, logits = od.prefill(m, x, [0, T], mask, round_fn=rnd)
        h2, logits2 = od.dense_forward(m, x, round_fn=rnd)
        tol = 1e-12 if rnd is od.identity else 1e-6
        np.testing.assert_allclose(h, h2, rtol=0, atol=tol * np.abs(h2).max())
        np.testing.assert_allclose(logits[0], logits2, rtol=0, atol=tol * np.abs(logits2).max())


def test_packed_sequences_are_independent():
    m, cfg = tiny_model(8)
    r = np.random.default_rng(9)
    xa = od.bf16_round(r.standard_normal((5, 256)))
    xb = od.bf16_round(r.standard_normal((7, 256)))
    zero = lambda T: np.zeros((2, T), dtype=np.uint8)
    ha, la = od.prefill(m, xa, [0, 5], zero(5))
    hb, lb = od.prefill(m, xb, [0, 7], zero(7))
    h, lg = od.prefill(m, np.concatenate([xa, xb]), [0, 5, 12], zero(12))
    np.testing.assert_allclose(h, np.concatenate([ha, hb]), rtol=0, atol=1e-12)
    np.testing.assert_allclose(lg, np.stack([la[0], lb[0]]), rtol=0, atol=1e-12)


def test_skipped_sublayer_is_identity_on_residual():
    m, cfg = tiny_model(10)
    T = 12
    x = od.bf16_round(np.random.default_rng(11).standard_normal((T, 256)))
    admit = np.array([-1, 0, 1, 0, -1, 1, 0, -1, -1, 0, 1, -1], dtype=np.int16)
    target = np.array([0, 1, 2, 2, 0, 1, 1, 0, 0, 2, 2, 0], dtype=np.uint8)
    mask = od.expand_adaptive_plan(admit, target, 2)
    trace = []
    od.prefill(m, x, [0, T], mask, trace=trace)
    before = [np.array(x, dtype=np.float64)] + trace[:-1]
    for l in range(2):
        for sub, bit in ((0, 1), (1, 2)):
            hin, hout = before[2 * l + sub], trace[2 * l + sub]
            skipped = (mask[l] & bit) != 0
            assert skipped.any()
            np.testing.assert_array_equal(hout[skipped], hin[skipped])
            assert np.abs(hout[~skipped] - hin[~skipped]).max() > 1e-3


def test_skip_attn_token_still_serves_as_key_and_value():
    cfg = dict(synth.TINY_DECODER, n_layers=1)
    m, cfg = tiny_model(12, cfg)
    T, j = 8, 3
    r = np.random.default_rng(13)
    x = od.bf16_round(r.standard_normal((T, 256)))
    mask = np.zeros((1, T), dtype=np.uint8)
    mask[0, j] = 1
    x2 = x.copy()
    x2[j] = od.bf16_round(x[j] + r.standard_normal(256))
    t1, t2 = [], []
    h1, _ = od.prefill(m, x, [0, T], mask, trace=t1)
    h2, _ = od.prefill(m, x2, [0, T], mask, trace=t2)
    np.testing.assert_array_equal(t1[0][j], x[j])                 # not a query, residual untouched
    np.testing.assert_array_equal(h1[:j], h2[:j])                 # causal: earlier tokens unaffected
    assert np.abs(t1[0][j + 1:] - t2[0][j + 1:]).max() > 1e-3     # later tokens read j's K/V


def test_plan_expansions():
    admit = np.array([-1, 0, 2, 3], dtype=np.int16)
    target = np.array([0, 1, 2, 1], dtype=np.uint8)
    m = od.expand_adaptive_plan(admit, target, 4)
    expect = np.array([[0, 1, 0, 0], [0, 1, 0, 0], [0, 1, 2, 0], [0, 1, 2, 1]], dtype=np.uint8)
    np.testing.assert_array_equal(m, expect)
    s = od.expand_static_plan([0, 2, 3], [1, 1, 0])
    np.testing.assert_array_equal(s, [[0, 0, 0], [2, 2, 0], [3, 3, 0]])


def test_projector_against_torch_layers():
    cfg = dict(synth.TINY_DECODER, d_vis=32, d_proj=48, d_model=256)
    w = synth.decoder_weights(14, cfg)
    m = od.model_from_torch(w, cfg)
    vis = od.bf16_round(np.random.default_rng(15).standard_normal((6, 32)))
    got = od.project(m, vis, round_fn=od.identity)
    t = torch.from_numpy(vis)
    hid = torch.nn.functional.gelu(t @ w["proj_w1"].double().T + w["proj_b1"].double())
    ref = hid @ w["proj_w2"].double().T + w["proj_b2"].double()
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_flop_model_reproduces_table1_vanilla_totals():
    # Table 1: LLaVA-1.5-7B vanilla 8.5 TFLOPs (576 visual + 64 text), LLaVA-NeXT-7B 42.7 TFLOPs.
    assert abs(flops.paper_prefill_flops(576 + 64) / 1e12 - 8.5) < 0.05
    assert abs(flops.paper_prefill_flops(2880 + 64) / 1e12 - 42.7) < 0.05


def test_table9_covers_every_layer_once():
    for name in synth.TABLE9:
        t = synth.TABLE9[name]
        assert sorted(t["attn"] + t["ffn"]) == list(range(32))
    assert (synth.skip_targets("llava-1.5-7b") == 2).sum() == 5
    assert (synth.skip_targets("llava-next-7b") == 2).sum() == 7


# ---- ASL-Skip online plan (§4.2, Eq. 6, Alg. 1 stage 2) -------------------------------------------
def test_normalized_entropy_closed_forms():
    np.testing.assert_allclose(od.normalized_entropy(np.zeros((2, 512))), 1.0, rtol=1e-14)
    one_hot = np.full((1, 100), -1e4)
    one_hot[0, 7] = 0.0
    assert od.normalized_entropy(one_hot)[0] < 1e-12
    two = np.full((1, 64), -1e4)
    two[0, :2] = 0.0  # two equally likely words: log 2 / log 64 = 1/6
    np.testing.assert_allclose(od.normalized_entropy(two), 1.0 / 6.0, rtol=1e-12)


def test_skippability_factors_and_clamp():
    model, _ = tiny_model(std=0.05)
    D = model["cfg"]["d_model"]
    rng = np.random.default_rng(3)
    q = rng.standard_normal(D)
    h = np.stack([q, -q, 2.0 * q, rng.standard_normal(D), q])  # rows 0-3 visual, 4 text
    seq_of = np.zeros(5, dtype=np.int64)
    s_sa, e, f = od.skippability(model, h, np.arange(4), seq_of, [np.array([4])])
    np.testing.assert_allclose(f[[0, 2]], 1.0, rtol=1e-12)  # parallel to the text mean
    np.testing.assert_allclose(f[1], 0.0, atol=1e-12)       # antiparallel
    assert np.all((e >= 0) & (e <= 1))
    np.testing.assert_allclose(s_sa, np.maximum(0.0, 1.0 - e - f), rtol=1e-15)
    assert s_sa[0] == 0.0 and s_sa[2] == 0.0  # F_itc = 1 leaves nothing to skip
    s0, _, f0 = od.skippability(model, h, np.arange(4), seq_of, [np.array([], dtype=np.int64)])
    np.testing.assert_allclose(f0, 0.5)  # no text in the sequence: cosine taken as 0


def _adaptive_case(n_layers=4, T=24, n_text=8):
    cfg = dict(synth.TINY_DECODER, n_layers=n_layers)
    model, _ = tiny_model(seed=9, cfg=cfg)
    x = od.bf16_round(np.random.default_rng(4).standard_normal((T, cfg["d_model"])))
    vis = np.r_[np.ones(T - n_text, bool), np.zeros(n_text, bool)]
    return model, x, vis


def test_adaptive_plan_with_w1_zero_admits_by_cumulative_slc():
    # without the online score every visual token is admitted at the first layer whose cumulative
    # w2 SLC^Norm reaches T_skip, with that layer's target; text tokens never
    model, x, vis = _adaptive_case()
    slc = np.array([0.3, 0.5, 0.4, 0.9])
    tgt = np.array([1, 2, 1, 2], np.uint8)
    _, _, admit, target, _ = od.prefill_adaptive(model, x, [0, len(x)], vis, slc, tgt, t_skip=0.75,
                                                 w1=0.0, w2=1.0, window=4)
    assert np.all(admit[vis] == 1) and np.all(target[vis] == 2)  # 0.3 + 0.5 >= 0.75 at layer 1
    assert np.all(admit[~vis] == -1)


def test_adaptive_plan_never_admitting_is_the_plain_prefill():
    model, x, vis = _adaptive_case()
    h, lg, admit, _, _ = od.prefill_adaptive(model, x, [0, len(x)], vis, np.ones(4), np.ones(4, np.uint8),
                                             t_skip=1e9, w1=3.0, w2=1.0, window=2)
    h0, lg0 = od.prefill(model, x, [0, len(x)], np.zeros((4, len(x)), np.uint8))
    assert np.all(admit == -1)
    np.testing.assert_array_equal(h, h0)
    np.testing.assert_array_equal(lg, lg0)


def test_adaptive_plan_equals_prefill_with_its_own_frozen_plan():
    # re-running the plain prefill with the plan the online rule produced gives the same stream:
    # the admission happens before the layer's forward and the target stays frozen
    model, x, vis = _adaptive_case(n_layers=6)
    slc = np.array([0.2, 0.9, 0.1, 0.6, 0.8, 0.3])
    tgt = np.array([1, 2, 2, 1, 1, 2], np.uint8)
    h, lg, admit, target, _ = od.prefill_adaptive(model, x, [0, len(x)], vis, slc, tgt, t_skip=1.0,
                                                  w1=3.0, w2=1.0, window=3)
    assert (admit >= 0).any()
    plan = od.expand_adaptive_plan(admit, target, 6)
    h0, lg0 = od.prefill(model, x, [0, len(x)], plan)
    np.testing.assert_array_equal(h, h0)
    np.testing.assert_array_equal(lg, lg0)
    assert np.all(admit < 3)  # decisions only inside the window


# ---- ablation variants of ASL-Skip (the ASL-Skip ablation table) ----------------------------------
def test_skippability_without_one_term():
    model, _ = tiny_model(std=0.05)
    D = model["cfg"]["d_model"]
    rng = np.random.default_rng(5)
    q = rng.standard_normal(D)
    h = np.stack([q, -q, np.zeros(D), q])  # rows 0-2 visual, 3 text
    seq_of = np.zeros(4, dtype=np.int64)
    # without E_ii: parallel to the text mean leaves nothing (F = 1), antiparallel everything (F = 0)
    s_sa, e, _ = od.skippability(model, h, np.arange(2), seq_of, [np.array([3])], use_entropy=False)
    np.testing.assert_array_equal(e, 0.0)
    np.testing.assert_allclose(s_sa, [0.0, 1.0], atol=1e-12)
    # without F_itc: a zero hidden state reads uniform logits through the lens (E = 1): S_sa = 0;
    # a one-hot vocabulary distribution would give S_sa = 1
    s_sa, _, f = od.skippability(model, h, np.array([2]), seq_of, [np.array([3])], use_itc=False)
    np.testing.assert_array_equal(f, 0.0)
    np.testing.assert_allclose(s_sa, [0.0], atol=1e-12)


def test_adaptive_plan_without_accumulation_needs_one_layer_over_threshold():
    # with w1 = 0, S_skip is w2 SLC^Norm(l) of the layer alone: the first layer whose own score
    # reaches T_skip (0.9 at layer 3), where accumulation admits at layer 1 (0.3 + 0.5)
    model, x, vis = _adaptive_case()
    slc = np.array([0.3, 0.5, 0.4, 0.9])
    tgt = np.array([1, 2, 1, 2], np.uint8)
    _, _, admit, target, _ = od.prefill_adaptive(model, x, [0, len(x)], vis, slc, tgt, t_skip=0.75,
                                                 w1=0.0, w2=1.0, window=4, accumulate=False)
    assert np.all(admit[vis] == 3) and np.all(target[vis] == 2)
    assert np.all(admit[~vis] == -1)


def test_adaptive_plan_without_slc_freezes_whole_layers():
    # without SLC an admitted token bypasses both sub-layers: its residual row stops changing at its
    # admission layer, so it equals the row that a run of only the layers before it leaves
    model, x, vis = _adaptive_case(n_layers=5)
    slc = np.full(5, 100.0)  # must have no effect
    tgt = np.array([1, 2, 1, 2, 1], np.uint8)
    kw = dict(t_skip=1.0, w1=1.0, w2=1.0, window=4, use_slc=False, use_entropy=False)
    h, _, admit, target, _ = od.prefill_adaptive(model, x, [0, len(x)], vis, slc, tgt, **kw)
    assert (admit > 0).any() and np.all(target[admit >= 0] == 3)
    for a in sorted(set(admit[admit > 0].tolist())):
        sub = dict(model, layers=model["layers"][:a], cfg=dict(model["cfg"], n_layers=a))
        h_a, _, admit_a, _, _ = od.prefill_adaptive(sub, x, [0, len(x)], vis, slc[:a], tgt[:a],
                                                   **dict(kw, window=min(4, a)))
        rows = np.flatnonzero(admit == a)
        np.testing.assert_array_equal(h[rows], h_a[rows])
        assert np.all(admit_a[rows] == -1)


def _torch_llama_forward(w, cfg, x):
    """One causal sequence through a LLaMA-style decoder written with torch.nn.functional in fp64:
    RMSNorm (F.rms_norm), rotate-half RoPE, scaled-dot-product attention with the causal mask and
    grouped K/V heads repeated per query group, SwiGLU as F.silu(y W_gate^T) * (y W_up^T). Shares
    nothing with the oracle but the weights."""
    F = torch.nn.functional
    H, Hkv, hd, eps, theta = (cfg[k] for k in ("n_heads", "n_kv_heads", "head_dim", "rms_eps",
                                                "rope_theta"))
    D = cfg["d_model"]
    f64 = lambda t: t.to(torch.float64)  # noqa: E731
    h = torch.as_tensor(x, dtype=torch.float64)
    T = h.shape[0]
    inv_freq = theta ** (-torch.arange(0, hd, 2, dtype=torch.float64) / hd)
    ang = torch.arange(T, dtype=torch.float64)[:, None] * inv_freq[None, :]
    cos, sin = torch.cat([ang.cos(), ang.cos()], -1), torch.cat([ang.sin(), ang.sin()], -1)

    def rotate_half(t):
        return torch.cat([-t[..., hd // 2:], t[..., :hd // 2]], -1)

    for lw in w["layers"]:
        xa = F.rms_norm(h, (D,), weight=f64(lw["attn_norm"]), eps=eps)
        q = (xa @ f64(lw["wq"]).T).view(T, H, hd).transpose(0, 1)
        k = (xa @ f64(lw["wk"]).T).view(T, Hkv, hd).transpose(0, 1)
        v = (xa @ f64(lw["wv"]).T).view(T, Hkv, hd).transpose(0, 1)
        q, k = q * cos + rotate_half(q) * sin, k * cos + rotate_half(k) * sin
        k, v = k.repeat_interleave(H // Hkv, dim=0), v.repeat_interleave(H // Hkv, dim=0)
        o = F.scaled_dot_product_attention(q[None], k[None], v[None], is_causal=True)[0]
        h = h + o.transpose(0, 1).reshape(T, H * hd) @ f64(lw["wo"]).T
        y = F.rms_norm(h, (D,), weight=f64(lw["ffn_norm"]), eps=eps)
        h = h + (F.silu(y @ f64(lw["w_gate"]).T) * (y @ f64(lw["w_up"]).T)) @ f64(lw["w_down"]).T
    z = F.rms_norm(h[-1:], (D,), weight=f64(w["final_norm"]), eps=eps)
    return h.numpy(), (z @ f64(w["lm_head"]).T)[0].numpy()


@pytest.mark.parametrize("kv_heads", [4, 2])
def test_prefill_equals_torch_functional_llama(kv_heads):
    # the oracle's decoder with an empty plan and no bf16 rounding against an independent torch
    # formulation of the same LLaMA-style layers (MHA and GQA), two packed sequences
    cfg = dict(n_layers=2, d_model=128, n_heads=4, n_kv_heads=kv_heads, head_dim=32, d_ffn=160,
               vocab=50, rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
    w = synth.decoder_weights(17, cfg, std=0.08)
    om = od.model_from_torch(w, cfg)
    x = np.random.default_rng(18).standard_normal((11, 128))
    cu = [0, 7, 11]
    h, lg = od.prefill(om, x, cu, np.zeros((2, 11), np.uint8), round_fn=od.identity)
    for b in range(2):
        h_t, lg_t = _torch_llama_forward(w, cfg, x[cu[b]:cu[b + 1]])
        np.testing.assert_allclose(h[cu[b]:cu[b + 1]], h_t, rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(lg[b], lg_t, rtol=1e-10, atol=1e-10)


def test_swiglu_gate_is_the_silu_operand():
    # swapping W_gate and W_up changes the layer (SiLU is not symmetric in its two factors), so the
    # comparison above fixes which weight the oracle gates
    cfg = dict(n_layers=1, d_model=64, n_heads=2, n_kv_heads=2, head_dim=32, d_ffn=96, vocab=10,
               rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
    w = synth.decoder_weights(19, cfg, std=0.2)
    om = od.model_from_torch(w, cfg)
    sw = od.model_from_torch(w, cfg)
    sw["layers"][0]["w_gate"], sw["layers"][0]["w_up"] = sw["layers"][0]["w_up"], sw["layers"][0]["w_gate"]
    x = np.random.default_rng(20).standard_normal((5, 64))
    h, _ = od.prefill(om, x, [0, 5], np.zeros((1, 5), np.uint8), round_fn=od.identity)
    hs, _ = od.prefill(sw, x, [0, 5], np.zeros((1, 5), np.uint8), round_fn=od.identity)
    h_t, _ = _torch_llama_forward(w, cfg, x)
    np.testing.assert_allclose(h, h_t, rtol=1e-10, atol=1e-10)
    assert np.abs(hs - h_t).max() > 1e-3
