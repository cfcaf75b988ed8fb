"""Helpers shared by the GPU parity tests (device marshalling and tolerance checks only)."""
import numpy as np
import torch

from oracle import prune as op
from paper_2609_34977_gb300 import _native as N
from paper_2609_34977_gb300 import synth


def bf16_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def rowwise_rel(g: np.ndarray, o: np.ndarray) -> float:
    """max over rows of max_j |g - o| / max_j |o|: the normwise reading of '2e-2 max relative'."""
    g = np.atleast_2d(g)
    o = np.atleast_2d(o)
    return float((np.abs(g - o).max(axis=1) / np.maximum(np.abs(o).max(axis=1), 1e-30)).max())


def conditioned_vision(seed0, n_tiles, n_patch, d, n_layers, n_heads, keep, final, *, has_cls=True,
                       attn_form=0, tries=64, **kw):
    """First seed from seed0 on whose tiles every discrete decision of the oracle has a margin
    above 1e-3 (see oracle.prune.well_conditioned). Returns (seed, inputs, oracle results)."""
    for seed in range(seed0, seed0 + tries):
        v = synth.vision_tiles(seed, n_tiles, n_patch, d, n_layers, n_heads, has_cls=has_cls,
                               attn_form=attn_form)
        res = op.prune(v["feats"], v["attn"], has_cls=has_cls, attn_form=attn_form,
                       final_layer=final, keep=keep, **kw)
        if all(op.well_conditioned(r) for r in res):
            return seed, v, res
    raise RuntimeError("no well-conditioned seed found")


def gpu_prune(v, keep, final, *, has_cls=True, attn_form=0, n_clusters=4, kmeans_iters=10,
              anchor_ratio=0.7, layer_weight=None, sim="cos", use_final_sim=True,
              use_anchor_sim=True):
    feats = [torch.from_numpy(f).cuda() for f in v["feats"]]
    attn = torch.from_numpy(v["attn"]).cuda()
    T, n_tok, d = feats[0].shape
    n = n_tok - (1 if has_cls else 0)
    cfg = N.prune_cfg(T, n_tok, d, len(feats), final, attn.shape[1], keep, has_cls=has_cls,
                      attn_form=attn_form, n_clusters=n_clusters, kmeans_iters=kmeans_iters,
                      anchor_ratio=anchor_ratio, layer_weight=layer_weight, sim=sim,
                      use_final_sim=use_final_sim, use_anchor_sim=use_anchor_sim)
    ws = torch.zeros(N.spd_prune_workspace_size(cfg), dtype=torch.uint8, device="cuda")
    keep_idx = torch.full((T, keep), -7, dtype=torch.int32, device="cuda")
    kind = torch.full((T, n), 9, dtype=torch.uint8, device="cuda")
    cluster = torch.full((T, n), 99, dtype=torch.int8, device="cuda")
    scores = torch.full((T, n), float("nan"), dtype=torch.float32, device="cuda")
    N.spd_prune(cfg, feats, attn, keep_idx, kind, cluster, scores, ws=ws)
    torch.cuda.synchronize()
    assert N.spd_workspace_status(ws) == 0
    return dict(keep_idx=keep_idx.cpu().numpy(), kind=kind.cpu().numpy(),
                cluster=cluster.cpu().numpy(), scores=scores.cpu().numpy(), feats=feats, ws=ws)


def assert_prune_parity(g, res, score_rtol=1e-5):
    for t, r in enumerate(res):
        np.testing.assert_array_equal(g["keep_idx"][t], r["keep_idx"])
        np.testing.assert_array_equal(g["kind"][t], r["kind"])
        np.testing.assert_array_equal(g["cluster"][t], r["cluster"])
        s_o = r["scores"]
        s_g = g["scores"][t].astype(np.float64)
        anchors = r["kind"] == 1
        assert np.isinf(s_g[anchors]).all()
        fin = ~anchors
        err = np.abs(s_g[fin] - s_o[fin]) / np.maximum(np.abs(s_o[fin]), 1e-2)
        if err.size:
            print(f"prune scores: max relative error {err.max():.3e} (tolerance {score_rtol:.0e})")
        assert err.max() <= score_rtol, err.max()
