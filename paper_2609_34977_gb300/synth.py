"""Seeded synthetic inputs shaped like the paper's workloads (§5.1 "Models", Table 1 shapes).

Both the CUDA path and the CPU oracle receive the same arrays from this module. It draws random
numbers with planted structure and holds none of the method's arithmetic: no scores, no selection,
no decoder math. The paper's benchmarks (GQA, MME, ...) and trained weights are not used; these
inputs stand in for their shapes only.

Recipe (vision side, one tile = one image or one AnyRes crop, §5.1 "Implementation Details"):

* Planted groups: patch i of a tile belongs to group z(i) = floor(i * G / n + 1/2) mod G, i.e.
  horizontal bands of the patch grid (background regions of an image), offset by half a band so
  that the K-means seeds (quantiles of the non-anchor tokens in index order) fall mid-band.
* Features of tapped layer l: F_l[i] = mu_{l,z(i)} + sigma_{l,i} * N(0, I_d), with group centres
  mu ~ 4 N(0, I_d) and per-token noise scales sigma ~ U(0.5, 3). The [CLS] row is N(0, I_d).
  The spread of sigma spreads the within-cluster similarity scores, which keeps selection cuts
  away from ties.
* Attention: per head, logits N(0, 2^2) over the (1 + n) columns, +2 on a salient quarter of the
  patches drawn uniformly (foreground concentration), then softmax over the row (CLS form), or over
  the n patches (received-attention form).

Decoder side: weights N(0, std^2) rounded to bf16, RMSNorm gains 1 + 0.2 N(0, 1) (gains far from 1
so that a dropped gain cannot go unnoticed), text embeddings N(0, 1) in bf16.

Skip plans follow Alg. 1: a fraction of the visual tokens enters skip mode at an admission layer
inside the decision window [0, L/2) and keeps the target m(admission layer) from Table 9.
"""
from __future__ import annotations

import math

import numpy as np

# Table 9 ("Replaced layers"): layer ids (0-based, each list covers 0..31 once) whose designated
# skip target m(l) is the attention or the FFN sub-layer.
TABLE9 = {
    "llava-1.5-7b": {
        "attn": (25, 27, 28, 30, 23, 26, 22, 24, 21, 0, 20, 3, 18, 4, 19, 17, 14, 15, 5, 16, 12, 1,
                 13, 7, 8, 9, 10),
        "ffn": (31, 29, 2, 11, 6),
    },
    "llava-next-7b": {
        "attn": (28, 29, 27, 30, 23, 24, 25, 22, 21, 26, 20, 19, 18, 17, 15, 16, 14, 12, 4, 13, 5, 0,
                 7, 6, 8),
        "ffn": (31, 1, 2, 3, 11, 9, 10),
    },
}

SKIP_ATTN = 1  # target codes of the adaptive plan, and mask bits of the expanded plan
SKIP_FFN = 2


def rng(seed: int) -> np.random.Generator:
    """Counter-based generator (Philox), identical on x86 and Arm hosts."""
    return np.random.Generator(np.random.Philox(int(seed)))


def skip_targets(model: str, n_layers: int = 32) -> np.ndarray:
    """m(l) for every decoder layer from Table 9, as SKIP_ATTN / SKIP_FFN codes."""
    tab = TABLE9[model]
    m = np.zeros(n_layers, dtype=np.uint8)
    for l in tab["attn"]:
        m[l] = SKIP_ATTN
    for l in tab["ffn"]:
        m[l] = SKIP_FFN
    assert (m > 0).all(), "Table 9 lists every layer once"
    return m


def seeded_skip_targets(seed: int, n_layers: int, ffn_share: float = 0.2) -> np.ndarray:
    """Stand-in m(l) for a decoder the paper has no Table 9 row for (Qwen2 shape)."""
    r = rng(seed)
    m = np.full(n_layers, SKIP_ATTN, dtype=np.uint8)
    m[r.random(n_layers) < ffn_share] = SKIP_FFN
    return m


def _salient_mask(r: np.random.Generator, n: int, frac: float = 0.25) -> np.ndarray:
    return r.random(n) < frac


def vision_tiles(seed: int, n_tiles: int, n_patch: int, d: int, n_layers: int, n_heads: int,
                 has_cls: bool = True, attn_form: int = 0, n_groups: int = 4):
    """Encoder features of `n_layers` tapped layers and one attention array per tile.

    Returns dict(feats=[float32 [n_tiles][n_tok][d]] * n_layers, attn=float32 [n_tiles][H][n_att],
    groups=int [n_tiles][n_patch]) where n_tok = n_patch + has_cls and n_att = n_tok for the CLS-row
    form (attn_form 0, column 0 is CLS->CLS) or n_patch for the received-attention form (1).
    """
    r = rng(seed)
    n_tok = n_patch + (1 if has_cls else 0)
    z = ((2 * np.arange(n_patch) * n_groups + n_patch) // (2 * n_patch)) % n_groups
    feats = [np.empty((n_tiles, n_tok, d), dtype=np.float32) for _ in range(n_layers)]
    n_att = n_tok if attn_form == 0 else n_patch
    attn = np.empty((n_tiles, n_heads, n_att), dtype=np.float32)
    groups = np.broadcast_to(z, (n_tiles, n_patch)).copy()
    for t in range(n_tiles):
        for l in range(n_layers):
            mu = 4.0 * r.standard_normal((n_groups, d))
            sigma = r.uniform(0.5, 3.0, size=n_patch)
            f = mu[z] + sigma[:, None] * r.standard_normal((n_patch, d))
            if has_cls:
                feats[l][t, 0] = r.standard_normal(d)
                feats[l][t, 1:] = f
            else:
                feats[l][t] = f
        sal = _salient_mask(r, n_patch)
        logits = 2.0 * r.standard_normal((n_heads, n_att))
        off = n_att - n_patch
        logits[:, off:] += 2.0 * sal[None, :]
        logits -= logits.max(axis=1, keepdims=True)
        e = np.exp(logits)
        attn[t] = (e / e.sum(axis=1, keepdims=True)).astype(np.float32)
    return dict(feats=feats, attn=attn, groups=groups)


def text_embeddings(seed: int, n_tokens: int, d_model: int) -> np.ndarray:
    """Text-token embeddings N(0,1), returned as bf16 bit patterns (uint16)."""
    import torch
    g = torch.Generator().manual_seed(int(seed))
    x = torch.randn(n_tokens, d_model, generator=g, dtype=torch.float32)
    return x.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def decoder_weights(seed: int, cfg: dict, std: float = 0.02, device: str = "cpu"):
    """Random-init bf16 weights of a LLaMA-style decoder (+ optional LLaVA MLP projector).

    cfg keys: n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn, vocab, d_vis, d_proj.
    Returns a dict of torch bf16 tensors on `device` (layers as a list of dicts). Matrices are
    [out_features][in_features] (row-major), as in y = x W^T.
    """
    import torch
    g = torch.Generator(device=device).manual_seed(int(seed))
    D, H, Hkv, hd, F = (cfg[k] for k in ("d_model", "n_heads", "n_kv_heads", "head_dim", "d_ffn"))

    def mat(o, i, s=std):
        return (torch.randn(o, i, generator=g, device=device) * s).to(torch.bfloat16)

    def gain(n):
        return (1.0 + 0.2 * torch.randn(n, generator=g, device=device)).to(torch.bfloat16)

    layers = []
    for _ in range(cfg["n_layers"]):
        layers.append(dict(attn_norm=gain(D), wq=mat(H * hd, D), wk=mat(Hkv * hd, D),
                           wv=mat(Hkv * hd, D), wo=mat(D, H * hd), ffn_norm=gain(D),
                           w_gate=mat(F, D), w_up=mat(F, D), w_down=mat(D, F)))
    w = dict(layers=layers, final_norm=gain(D), lm_head=mat(cfg["vocab"], D))
    if cfg.get("d_proj", 0):
        dv, dp = cfg["d_vis"], cfg["d_proj"]
        w["proj_w1"] = mat(dp, dv, 1.0 / math.sqrt(dv))
        w["proj_b1"] = (0.1 * torch.randn(dp, generator=g, device=device)).to(torch.bfloat16)
        w["proj_w2"] = mat(D, dp, 1.0 / math.sqrt(dp))
        w["proj_b2"] = (0.1 * torch.randn(D, generator=g, device=device)).to(torch.bfloat16)
    return w


def adaptive_plan(seed: int, n_layers: int, token_is_visual: np.ndarray, skip_frac: float,
                  m: np.ndarray, admit_lo: int = 0, admit_hi: int | None = None):
    """Per-token (admission layer, frozen target) pairs in the form Alg. 1 produces.

    A fraction `skip_frac` of the visual tokens enters skip mode; its admission layer is drawn
    uniformly from [admit_lo, admit_hi) inside the decision window l < L/2, and its target is
    m(admission layer). Text tokens never enter skip mode. admit = -1 means never.
    """
    r = rng(seed)
    if admit_hi is None:
        admit_hi = n_layers // 2
    T = len(token_is_visual)
    admit = np.full(T, -1, dtype=np.int16)
    target = np.zeros(T, dtype=np.uint8)
    vis = np.flatnonzero(token_is_visual)
    chosen = vis[r.random(len(vis)) < skip_frac]
    e = r.integers(admit_lo, admit_hi, size=len(chosen))
    admit[chosen] = e
    target[chosen] = m[e]
    return admit, target


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns (uint16) to float32."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# --- workload shapes (the paper's models, §5.1 and Table 1) ---------------------------------
TINY_DECODER = dict(n_layers=2, d_model=256, n_heads=4, n_kv_heads=4, head_dim=64, d_ffn=688,
                    vocab=512, rope_theta=1e4, rms_eps=1e-5, d_vis=0, d_proj=0)
LLAVA_7B_DECODER = dict(n_layers=32, d_model=4096, n_heads=32, n_kv_heads=32, head_dim=128,
                        d_ffn=11008, vocab=32000, rope_theta=1e4, rms_eps=1e-5, d_vis=1024,
                        d_proj=4096)
QWEN2_DECODER = dict(n_layers=28, d_model=3584, n_heads=28, n_kv_heads=4, head_dim=128,
                     d_ffn=18944, vocab=152064, rope_theta=1e6, rms_eps=1e-6, d_vis=1280,
                     d_proj=3584)
