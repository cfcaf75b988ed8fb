"""CPU oracle of the decoder prefill with adaptive sub-layer skipping (§4.2, §4.3, Alg. 1 stage 2).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import
this module. It shares no code with the CUDA path.

The paper does not describe the decoder beyond its attention and FFN sub-layers. The architecture
is LLaMA-style, from the models it evaluates (LLaVA-1.5/NeXT on Vicuna-7B, Qwen2-style decoders):
RMSNorm, rotary position embedding (rotate-half), causal multi-head or grouped-query attention,
SwiGLU FFN, no biases. LLaVA's projector is Linear-GELU-Linear with biases.

Skipping (§3.2, Alg. 1):
* VSkip-Attn: the token is not a query, and its residual is not updated by attention. It still acts
  as a key and a value for every other token.
* VSkip-FFN: the token's FFN update is bypassed (residual identity).
The plan is per layer and per token: bit 1 = skip attention, bit 2 = skip FFN.

Precision: fp64 arithmetic. Values are rounded to bf16 (round to nearest even) where the GPU path
stores bf16: norm outputs, Q/K/V after rotary embedding, the attention output, the SwiGLU product,
and the projector's hidden and output rows. Pass round_fn=identity for pure fp64.
"""
from __future__ import annotations

import numpy as np


def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round to the nearest bfloat16 value (8 significant bits), ties to even, kept in float64."""
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)                  # x = m * 2^e, 0.5 <= |m| < 1
    return np.ldexp(np.round(m * 256.0) / 256.0, e)


def identity(x):
    return np.asarray(x, dtype=np.float64)


def rmsnorm(h: np.ndarray, gain: np.ndarray, eps: float) -> np.ndarray:
    """gain * h / sqrt(mean(h^2) + eps), row by row."""
    h = np.asarray(h, dtype=np.float64)
    return gain * h / np.sqrt((h * h).mean(axis=-1, keepdims=True) + eps)


def rope(x: np.ndarray, pos: np.ndarray, n_heads: int, head_dim: int, theta: float) -> np.ndarray:
    """Rotary position embedding, rotate-half form, on rows x [T][n_heads * head_dim].

    Pair (j, j + head_dim/2) of every head is rotated by the angle pos * theta^(-2j/head_dim).
    """
    half = head_dim // 2
    inv = theta ** (-(2.0 * np.arange(half)) / head_dim)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    xh = np.asarray(x, dtype=np.float64).reshape(len(x), n_heads, head_dim)
    x1, x2 = xh[..., :half], xh[..., half:]
    out = np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)
    return out.reshape(len(x), n_heads * head_dim)


def causal_attention(q, k, v, q_pos, k_pos, n_heads, n_kv_heads, head_dim):
    """softmax(q k^T / sqrt(head_dim)) v for one sequence, a query seeing keys with k_pos <= q_pos.

    q: [Tq][H*hd] for any subset of the sequence's tokens (with their positions q_pos); k, v:
    [Tk][Hkv*hd] for every token of the sequence. Query head h reads key/value head
    h // (H / Hkv).
    """
    grp = n_heads // n_kv_heads
    out = np.zeros((len(q), n_heads * head_dim))
    allowed = np.asarray(k_pos)[None, :] <= np.asarray(q_pos)[:, None]
    for h in range(n_heads):
        kh = h // grp
        qh = q[:, h * head_dim:(h + 1) * head_dim]
        kk = k[:, kh * head_dim:(kh + 1) * head_dim]
        vv = v[:, kh * head_dim:(kh + 1) * head_dim]
        s = (qh @ kk.T) / np.sqrt(head_dim)
        s = np.where(allowed, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p /= p.sum(axis=1, keepdims=True)
        out[:, h * head_dim:(h + 1) * head_dim] = p @ vv
    return out


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu(x):
    """Exact (erf) GELU, as in LLaVA's mlp2x_gelu projector."""
    from scipy.special import erf
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def project(model, vis, round_fn=bf16_round):
    """LLaVA MLP projector (the connector of §2): Linear(d_vis->d_proj)+GELU, Linear(->D)."""
    p = model["proj"]
    hid = round_fn(gelu(np.asarray(vis, dtype=np.float64) @ p["w1"].T + p["b1"]))
    return round_fn(hid @ p["w2"].T + p["b2"])


def expand_adaptive_plan(admit, target, n_layers):
    """Per-layer skip bits of Alg. 1's frozen-target plan.

    Token i enters skip mode at layer admit[i] (-1 = never) and from that layer on (Alg. 1 admits
    before the layer's forward) bypasses the sub-layer target[i] (1 attention, 2 FFN).
    """
    admit = np.asarray(admit, dtype=np.int64)
    mask = np.zeros((n_layers, len(admit)), dtype=np.uint8)
    for i in range(len(admit)):
        if admit[i] >= 0:
            mask[admit[i]:, i] = target[i]
    return mask


def expand_static_plan(layer_mask, token_sel):
    """Static sparse-layer replacement (§3.2): layer l replaces the sub-layers in layer_mask[l]
    (bits as above) by VSkip layers for every selected token (the visual tokens)."""
    layer_mask = np.asarray(layer_mask, dtype=np.uint8)
    token_sel = np.asarray(token_sel, dtype=bool)
    return (layer_mask[:, None] * token_sel[None, :]).astype(np.uint8)


def forward_layer(cfg, w, h, mask_l, cu, pos, round_fn=bf16_round, trace=None):
    """One decoder layer in place on the residual stream h [T][D]: tokens with bit 0 of mask_l
    bypass attention (not queries; still keys and values), tokens with bit 1 bypass the FFN."""
    H, Hkv, hd, eps = cfg["n_heads"], cfg["n_kv_heads"], cfg["head_dim"], cfg["rms_eps"]
    xa = round_fn(rmsnorm(h, w["attn_norm"], eps))
    k = round_fn(rope(xa @ w["wk"].T, pos, Hkv, hd, cfg["rope_theta"]))
    v = round_fn(xa @ w["wv"].T)
    act = np.flatnonzero((mask_l & 1) == 0)
    if len(act):
        q = round_fn(rope(xa[act] @ w["wq"].T, pos[act], H, hd, cfg["rope_theta"]))
        o = np.zeros((len(act), H * hd))
        for b in range(len(cu) - 1):
            rows = np.flatnonzero((act >= cu[b]) & (act < cu[b + 1]))
            if len(rows):
                sl = slice(cu[b], cu[b + 1])
                o[rows] = causal_attention(q[rows], k[sl], v[sl], pos[act[rows]], pos[sl],
                                           H, Hkv, hd)
        h[act] += round_fn(o) @ w["wo"].T
    if trace is not None:
        trace.append(h.copy())
    actf = np.flatnonzero((mask_l & 2) == 0)
    if len(actf):
        y = round_fn(rmsnorm(h[actf], w["ffn_norm"], eps))
        a = round_fn(silu(y @ w["w_gate"].T) * (y @ w["w_up"].T))
        h[actf] += a @ w["w_down"].T
    if trace is not None:
        trace.append(h.copy())


def prefill(model, x, cu_seqlens, skip_mask, round_fn=bf16_round, trace=None):
    """Decoder prefill over packed sequences with per-layer, per-token sub-layer bypass.

    x: [T][D] input embeddings (bf16 values). cu_seqlens: sequence boundaries [B+1]. skip_mask:
    [L][T]. Returns (h [T][D] final residual stream, logits [B][V] of each sequence's last token).
    If `trace` is a list, the residual stream after every sub-layer is appended to it.
    """
    cfg = model["cfg"]
    h = np.array(x, dtype=np.float64)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    pos = np.concatenate([np.arange(cu[b + 1] - cu[b]) for b in range(len(cu) - 1)])
    for l, w in enumerate(model["layers"]):
        forward_layer(cfg, w, h, skip_mask[l], cu, pos, round_fn, trace)
    last = cu[1:] - 1
    z = round_fn(rmsnorm(h[last], model["final_norm"], cfg["rms_eps"]))
    return h, z @ model["lm_head"].T


def normalized_entropy(logits):
    """Shannon entropy of softmax(logits) per row divided by log V (§4.2.1 E_ii in [0, 1])."""
    z = np.asarray(logits, dtype=np.float64)
    z = z - z.max(axis=-1, keepdims=True)
    p = np.exp(z)
    p /= p.sum(axis=-1, keepdims=True)
    plogp = np.where(p > 0, p * np.log(np.where(p > 0, p, 1.0)), 0.0)
    return -plogp.sum(axis=-1) / np.log(z.shape[-1])


def skippability(model, h, cand, seq_of, text_rows, round_fn=bf16_round, use_entropy=True,
                 use_itc=True):
    """S_sa(i, l) = ReLU(1 - E_ii - F_itc) for the candidate tokens (§4.2.1).

    E_ii: normalized entropy of the vocabulary distribution of the token's hidden state, read
    through the unembedding after the final RMSNorm (the logit-lens reading; the operand rounded to
    bf16 as every GEMM input). F_itc = (cos(h_i, q_t) + 1) / 2 with q_t the mean hidden state of the
    text tokens of the token's sequence (cos = 0 when that sequence has no text tokens).
    use_entropy / use_itc False: the ablations of S_sa's components (ASL-Skip ablation table,
    part (c)); the dropped term is left out of the sum (reading), and is returned as 0.
    """
    cfg = model["cfg"]
    e = np.zeros(len(cand))
    if use_entropy:
        z = round_fn(rmsnorm(h[cand], model["final_norm"], cfg["rms_eps"]))
        e = normalized_entropy(z @ model["lm_head"].T)
    f = np.zeros(len(cand))
    for n, i in enumerate(cand):
        if not use_itc:
            continue
        t = text_rows[seq_of[i]]
        if len(t) == 0:
            f[n] = 0.5
            continue
        q = h[t].mean(axis=0)
        den = np.linalg.norm(h[i]) * np.linalg.norm(q)
        f[n] = ((h[i] @ q) / den if den > 0 else 0.0) * 0.5 + 0.5
    return np.maximum(0.0, 1.0 - e - f), e, f


def prefill_adaptive(model, x, cu_seqlens, is_visual, slc_norm, layer_target, t_skip, w1, w2,
                     window, round_fn=bf16_round, use_entropy=True, use_itc=True, accumulate=True,
                     use_slc=True):
    """Alg. 1 stage 2 with the online plan: at each layer l < window, every visual token not yet
    in skip mode accumulates S_skip += w1 S_sa(i, l) + w2 SLC^Norm(l) (Eq. 6); once S_skip >= T_skip
    it enters skip mode with target m(l) = layer_target[l], frozen, and bypasses that sub-layer
    from layer l on. Returns (h, logits, admit [T] (-1 never), target [T], margin), margin = the
    smallest |S_skip - T_skip| over every comparison made (for choosing well-conditioned tests).

    Ablations of the ASL-Skip table: w1 = 0 (without S_sa); use_entropy / use_itc False (without
    E_ii / F_itc, see skippability); accumulate False (S_skip is the current layer's S_fuse alone);
    use_slc False (no w2 SLC^Norm term, and an admitted token bypasses both sub-layers: whole
    layers, the paper's description of that variant).
    """
    cfg = model["cfg"]
    L = cfg["n_layers"]
    h = np.array(x, dtype=np.float64)
    T = len(h)
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    pos = np.concatenate([np.arange(cu[b + 1] - cu[b]) for b in range(len(cu) - 1)])
    seq_of = np.concatenate([np.full(cu[b + 1] - cu[b], b) for b in range(len(cu) - 1)])
    vis = np.asarray(is_visual, dtype=bool)
    text_rows = [np.flatnonzero((seq_of == b) & ~vis) for b in range(len(cu) - 1)]
    admit = np.full(T, -1, dtype=np.int64)
    target = np.zeros(T, dtype=np.uint8)
    s_skip = np.zeros(T)
    margin = np.inf
    for l in range(L):
        if l < window:
            cand = np.flatnonzero(vis & (admit < 0))
            if len(cand):
                s_sa, _, _ = skippability(model, h, cand, seq_of, text_rows, round_fn,
                                          use_entropy, use_itc)
                s_fuse = w1 * s_sa + (w2 * slc_norm[l] if use_slc else 0.0)
                s_skip[cand] = (s_skip[cand] + s_fuse) if accumulate else s_fuse
                margin = min(margin, float(np.abs(s_skip[cand] - t_skip).min()))
                new = cand[s_skip[cand] >= t_skip]
                admit[new] = l
                target[new] = layer_target[l] if use_slc else 3
        mask_l = np.where((admit >= 0) & (admit <= l), target, 0).astype(np.uint8)
        forward_layer(cfg, model["layers"][l], h, mask_l, cu, pos, round_fn)
    last = cu[1:] - 1
    z = round_fn(rmsnorm(h[last], model["final_norm"], cfg["rms_eps"]))
    return h, z @ model["lm_head"].T, admit, target, margin


def dense_forward(model, x, round_fn=bf16_round):
    """Textbook causal LLaMA-style forward of ONE sequence, token by token and head by head.

    Written independently of prefill() (no row lists, no packing) so that prefill() with an
    all-zero plan can be checked against it. Returns (h [T][D], logits of the last token [V]).
    """
    cfg = model["cfg"]
    H, Hkv, hd, eps, theta = (cfg[k] for k in ("n_heads", "n_kv_heads", "head_dim", "rms_eps",
                                                "rope_theta"))
    h = np.array(x, dtype=np.float64)
    T, D = h.shape
    half = hd // 2

    def rot(vec, p):
        out = vec.copy()
        for j in range(half):
            a = p * theta ** (-2.0 * j / hd)
            out[j] = vec[j] * np.cos(a) - vec[j + half] * np.sin(a)
            out[j + half] = vec[j + half] * np.cos(a) + vec[j] * np.sin(a)
        return out

    for w in model["layers"]:
        keys, vals, queries = [], [], []
        for t in range(T):
            xt = round_fn(w["attn_norm"] * h[t] / np.sqrt(np.mean(h[t] ** 2) + eps))
            qt = xt @ w["wq"].T
            kt = xt @ w["wk"].T
            queries.append(round_fn(np.concatenate([rot(qt[i * hd:(i + 1) * hd], t) for i in range(H)])))
            keys.append(round_fn(np.concatenate([rot(kt[i * hd:(i + 1) * hd], t) for i in range(Hkv)])))
            vals.append(round_fn(xt @ w["wv"].T))
        attn_out = np.zeros((T, H * hd))
        for t in range(T):
            for i in range(H):
                j = i * Hkv // H
                sc = np.array([queries[t][i * hd:(i + 1) * hd] @ keys[u][j * hd:(j + 1) * hd]
                               for u in range(t + 1)]) / np.sqrt(hd)
                pr = np.exp(sc - sc.max())
                pr /= pr.sum()
                attn_out[t, i * hd:(i + 1) * hd] = sum(pr[u] * vals[u][j * hd:(j + 1) * hd]
                                                       for u in range(t + 1))
        for t in range(T):
            h[t] = h[t] + round_fn(attn_out[t]) @ w["wo"].T
        for t in range(T):
            yt = round_fn(w["ffn_norm"] * h[t] / np.sqrt(np.mean(h[t] ** 2) + eps))
            g = yt @ w["w_gate"].T
            u = yt @ w["w_up"].T
            h[t] = h[t] + round_fn(g / (1.0 + np.exp(-g)) * u) @ w["w_down"].T
    zt = round_fn(model["final_norm"] * h[-1] / np.sqrt(np.mean(h[-1] ** 2) + eps))
    return h, zt @ model["lm_head"].T


def model_from_torch(w: dict, cfg: dict) -> dict:
    """float64 numpy copy of a weight dict of torch bf16 tensors (as drawn by synth)."""
    def f(t):
        return t.detach().to("cpu").float().numpy().astype(np.float64)
    m = dict(cfg=dict(cfg), layers=[{k: f(v) for k, v in lw.items()} for lw in w["layers"]],
             final_norm=f(w["final_norm"]), lm_head=f(w["lm_head"]))
    if "proj_w1" in w:
        m["proj"] = dict(w1=f(w["proj_w1"]), b1=f(w["proj_b1"]), w2=f(w["proj_w2"]),
                         b2=f(w["proj_b2"]))
    return m
