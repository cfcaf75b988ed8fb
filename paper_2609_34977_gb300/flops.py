"""Work accounting for the prefill: the paper's FLOP convention and the algorithmic flops/bytes of
each step, used for throughput and roofline fractions.

Paper convention (Table 1 TFLOPs column): per decoder layer 4 n d^2 + 2 n^2 d + 3 n d m
multiply-adds, i.e. 2 * L * (4 n d^2 + 2 n^2 d + 3 n d m) FLOPs for n tokens (visual + text),
hidden d, FFN width m. With n = 576 + 64 it gives 8.5 TFLOPs for LLaVA-1.5-7B, and with
n = 2880 + 64 it gives 42.7 TFLOPs for LLaVA-NeXT-7B (Table 1, vanilla rows).
"""
from __future__ import annotations

import numpy as np


def paper_prefill_flops(n_tokens: int, n_layers: int = 32, d: int = 4096, m: int = 11008) -> float:
    """Vanilla prefill FLOPs in the paper's Table 1 convention."""
    n = float(n_tokens)
    return 2.0 * n_layers * (4 * n * d * d + 2 * n * n * d + 3 * n * d * m)


def prefill_work(cfg: dict, seq_lens, skip_mask: np.ndarray, n_proj_rows: int = 0):
    """Algorithmic FLOPs and weight bytes of one skip-aware prefill as this library executes it.

    Per layer: K/V projections over every token; Q, attention and the output projection over the
    attention-active tokens; gate/up/down over the FFN-active tokens; then the LM head on the last
    token of each sequence and the projector on the visual rows. Attention counts the causal
    context of each active query (2 * ctx * hd for QK^T and again for PV, per head).
    Returns dict(gemm_flops, attn_flops, weight_bytes, per_layer=[...]).
    """
    D, H, Hkv, hd, F, V = (cfg[k] for k in ("d_model", "n_heads", "n_kv_heads", "head_dim",
                                            "d_ffn", "vocab"))
    T = int(sum(seq_lens))
    pos = np.concatenate([np.arange(s) for s in seq_lens])
    gemm = attn = 0.0
    wbytes = 0.0
    per_layer = []
    for l in range(cfg["n_layers"]):
        a = (skip_mask[l] & 1) == 0
        f = (skip_mask[l] & 2) == 0
        ta, tf = int(a.sum()), int(f.sum())
        g = 2.0 * T * D * 2 * Hkv * hd + 2.0 * ta * D * H * hd * 2 + 2.0 * tf * D * F * 3
        at = 4.0 * H * hd * float((pos[a] + 1).sum())
        wb = 2.0 * D * 2 * Hkv * hd + (2.0 * D * H * hd * 2 if ta else 0) + (2.0 * 3 * D * F if tf else 0)
        per_layer.append(dict(attn_rows=ta, ffn_rows=tf, gemm_flops=g, attn_flops=at))
        gemm += g
        attn += at
        wbytes += wb
    B = len(seq_lens)
    gemm += 2.0 * B * D * V
    wbytes += 2.0 * D * V
    if n_proj_rows and cfg.get("d_proj"):
        gemm += 2.0 * n_proj_rows * (cfg["d_vis"] * cfg["d_proj"] + cfg["d_proj"] * D)
        wbytes += 2.0 * (cfg["d_vis"] * cfg["d_proj"] + cfg["d_proj"] * D)
    return dict(gemm_flops=gemm, attn_flops=attn, weight_bytes=wbytes, per_layer=per_layer)


def prune_bytes(n_tiles: int, n_tok: int, d: int, n_layers: int, n_heads: int, n_att: int,
                keep: int) -> float:
    """Algorithmic HBM bytes of pruning a batch of tiles: every tapped layer's features read once,
    the attention rows read once, the kept indices written, and the kept payload rows read (fp32)
    and written (bf16)."""
    return n_tiles * (n_layers * n_tok * d * 4.0 + n_heads * n_att * 4.0 + keep * (4.0 + d * 6.0))
