"""One SPIDER prefill step (Alg. 1) over a batch of requests, as a sequence of libspider.so calls.

This module only owns buffers and workspaces and calls the C ABI in order. Every computation runs
in the CUDA library:

    spd_prune              MSV-Prune of every tile (Sec. 4.1)
    spd_gather_rows_bf16   kept final-layer rows -> bf16
    spd_project            LLaVA projector into the decoder input rows (or a row copy when the
                           vision width equals the decoder width and no projector is configured)
    spd_scatter_rows       text embeddings into their rows
    spd_prefill            decoder prefill with the per-layer, per-token skip mask (Sec. 4.2-4.3)
    spd_prefill_adaptive   ... or with the skip plan computed online (Alg. 1 stage 2)

Sequence layout per request: [kept visual tokens of its tiles, in tile order and spatial order;
text tokens]. Alg. 1 writes the text first; the order is a layout choice of the caller and the
decoder treats both the same way.
"""
from __future__ import annotations

import numpy as np
import torch

from . import _native as N


class SpiderPrefill:
    """Buffers and workspaces for a fixed batch layout.

    tiles_per_req[b] tiles and text_lens[b] text tokens for request b; `keep` tokens kept per tile
    skip_mask [L][T] host uint8 or None. dense=True is the un-pruned baseline: every patch is kept
    in order (no MSV-Prune call) and the same gather/projector/decoder kernels run.
    """

    def __init__(self, model: N.SpdModel, *, n_patch: int, has_cls: bool, d_vis: int,
                 n_feat_layers: int, final_layer: int, n_heads_vis: int, attn_form: int,
                 keep: int, tiles_per_req, text_lens, n_clusters: int = 4, kmeans_iters: int = 10,
                 anchor_ratio: float = 0.7, layer_weight=None, dense: bool = False,
                 device: str = "cuda"):
        self.model = model
        cfg = model.cfg
        self.D = cfg["d_model"]
        self.tiles_per_req = list(tiles_per_req)
        self.text_lens = list(text_lens)
        self.n_tiles = int(sum(self.tiles_per_req))
        self.dense = dense
        if dense:
            keep = n_patch
        self.keep = keep
        self.n_patch = n_patch
        self.n_tok = n_patch + (1 if has_cls else 0)
        self.d_vis = d_vis
        self.B = len(self.text_lens)
        self.prune_cfg = N.prune_cfg(self.n_tiles, self.n_tok, d_vis, n_feat_layers, final_layer,
                                     n_heads_vis, keep, has_cls=has_cls, attn_form=attn_form,
                                     n_clusters=n_clusters, kmeans_iters=kmeans_iters,
                                     anchor_ratio=anchor_ratio, layer_weight=layer_weight)
        self.has_projector = bool(cfg.get("d_proj"))
        if not self.has_projector and d_vis != self.D:
            raise ValueError("without a projector the vision width must equal d_model")
        # sequence layout
        vis_rows, text_rows, cu = [], [], [0]
        row = 0
        for b in range(self.B):
            nv = self.tiles_per_req[b] * keep
            vis_rows.extend(range(row, row + nv))
            row += nv
            text_rows.extend(range(row, row + self.text_lens[b]))
            row += self.text_lens[b]
            cu.append(row)
        self.T = row
        self.cu = np.array(cu, dtype=np.int32)
        self.token_is_visual = np.zeros(self.T, dtype=bool)
        self.token_is_visual[vis_rows] = True
        dev = torch.device(device)
        self.vis_rows = torch.tensor(vis_rows, dtype=torch.int32, device=dev)
        self.text_rows = torch.tensor(text_rows, dtype=torch.int32, device=dev)
        # buffers
        self.keep_idx = torch.empty(self.n_tiles, keep, dtype=torch.int32, device=dev)
        if dense:
            self.keep_idx.copy_(torch.arange(keep, dtype=torch.int32, device=dev).expand(self.n_tiles, keep))
        self.vis = torch.empty(self.n_tiles * keep, d_vis, dtype=torch.bfloat16, device=dev)
        self.x = torch.empty(self.T, self.D, dtype=torch.bfloat16, device=dev)
        self.h = torch.empty(self.T, self.D, dtype=torch.float32, device=dev)
        self.logits = torch.empty(self.B, cfg["vocab"], dtype=torch.float32, device=dev)
        self.ws_prune = torch.zeros(N.spd_prune_workspace_size(self.prune_cfg), dtype=torch.uint8,
                                    device=dev)
        self.ws_proj = (torch.zeros(N.spd_project_workspace_size(model, self.n_tiles * keep),
                                    dtype=torch.uint8, device=dev) if self.has_projector else None)
        self.ws_prefill = torch.zeros(N.spd_prefill_workspace_size(model, self.T, self.B),
                                      dtype=torch.uint8, device=dev)
        self.ws_adaptive = None
        self.admit = None

    def run(self, feats, attn, text, skip_mask, stream=None, policy=None):
        """Enqueue one step on device inputs: feats (list of [n_tiles][n_tok][d_vis] fp32), attn,
        text [sum(text_lens)][D] bf16. Returns the logits tensor [B][vocab] (device).

        policy (dict: slc_norm, layer_target, t_skip, w1, w2, window, optional ablate bits
        SPD_SKIP_NO_* and device_plan) replaces skip_mask by the online ASL-Skip plan; the admission layer of every
        token is then left in self.admit."""
        if not self.dense:
            N.spd_prune(self.prune_cfg, feats, attn, self.keep_idx, ws=self.ws_prune, stream=stream)
        fin = int(self.prune_cfg.final_layer)
        N.spd_gather_rows_bf16(feats[fin], self.n_tiles, self.n_tok, self.d_vis,
                               1 if self.prune_cfg.has_cls else 0, self.keep_idx, self.keep, self.vis,
                               ws=self.ws_prune, stream=stream)
        nv = self.n_tiles * self.keep
        if self.has_projector:
            N.spd_project(self.model, self.vis, nv, self.vis_rows, self.x, self.ws_proj, stream=stream)
        else:
            N.spd_scatter_rows(self.model, self.vis, nv, self.vis_rows, self.x, stream=stream)
        if len(self.text_rows):
            N.spd_scatter_rows(self.model, text, len(self.text_rows), self.text_rows, self.x,
                               stream=stream)
        if policy is None:
            N.spd_prefill(self.model, self.x, self.T, self.cu, skip_mask, self.h, self.logits,
                          self.ws_prefill, stream=stream)
            return self.logits
        if self.ws_adaptive is None:
            self.ws_adaptive = torch.zeros(N.spd_prefill_adaptive_workspace_size(self.model, self.T, self.B),
                                           dtype=torch.uint8, device=self.h.device)
        self.admit = N.spd_prefill_adaptive(self.model, self.x, self.T, self.cu, self.token_is_visual,
                                            policy["slc_norm"], policy["layer_target"], policy["t_skip"],
                                            policy["w1"], policy["w2"], policy["window"], self.h,
                                            self.logits, self.ws_adaptive, stream=stream,
                                            ablate=policy.get("ablate", 0),
                                            device_plan=policy.get("device_plan", 0))
        return self.logits

    def status(self) -> int:
        """First device-side failure recorded by any call of this pipeline (0 = none)."""
        codes = [N.spd_workspace_status(w) for w in (self.ws_prune, self.ws_proj, self.ws_prefill,
                                                     self.ws_adaptive) if w is not None]
        return next((c for c in codes if c), 0)


class VarResSpiderPrefill:
    """One image per request with its own token count (dynamic resolution, e.g. the Qwen2-VL
    encoder after its 2 x 2 patch merger: no [CLS] token, so the received-attention form of
    Sec. 4.1.1), pruned to round(keep_ratio * n_i) tokens each; then the projector, the sequence
    assembly [visual; text] per request and the decoder prefill, as in SpiderPrefill.

    n_patches[b] tokens in image b (its own spd_prune call); dense=True keeps every token."""

    def __init__(self, model: N.SpdModel, *, n_patches, d_vis: int, n_feat_layers: int,
                 final_layer: int, n_heads_vis: int, keep_ratio: float, text_lens,
                 n_clusters: int = 4, kmeans_iters: int = 10, anchor_ratio: float = 0.7,
                 dense: bool = False, device: str = "cuda"):
        self.model = model
        cfg = model.cfg
        self.D = cfg["d_model"]
        self.n_patches = [int(n) for n in n_patches]
        self.text_lens = list(text_lens)
        self.B = len(self.n_patches)
        self.dense = dense
        self.d_vis = d_vis
        self.final_layer = final_layer
        self.keeps = [n if dense else max(1, int(round(keep_ratio * n))) for n in self.n_patches]
        self.cfgs = [N.prune_cfg(1, n, d_vis, n_feat_layers, final_layer, n_heads_vis, k, has_cls=False,
                                 attn_form=1, n_clusters=n_clusters, kmeans_iters=kmeans_iters,
                                 anchor_ratio=anchor_ratio)
                     for n, k in zip(self.n_patches, self.keeps)]
        dev = torch.device(device)
        vis_rows, text_rows, cu = [], [], [0]
        row = 0
        for b in range(self.B):
            vis_rows.extend(range(row, row + self.keeps[b]))
            row += self.keeps[b]
            text_rows.extend(range(row, row + self.text_lens[b]))
            row += self.text_lens[b]
            cu.append(row)
        self.T = row
        self.cu = np.array(cu, dtype=np.int32)
        self.token_is_visual = np.zeros(self.T, dtype=bool)
        self.token_is_visual[vis_rows] = True
        self.vis_rows = torch.tensor(vis_rows, dtype=torch.int32, device=dev)
        self.text_rows = torch.tensor(text_rows, dtype=torch.int32, device=dev)
        self.keep_idx = [torch.arange(k, dtype=torch.int32, device=dev) if dense else
                         torch.empty(k, dtype=torch.int32, device=dev) for k in self.keeps]
        nv = sum(self.keeps)
        self.vis = torch.empty(nv, d_vis, dtype=torch.bfloat16, device=dev)
        self.x = torch.empty(self.T, self.D, dtype=torch.bfloat16, device=dev)
        self.h = torch.empty(self.T, self.D, dtype=torch.float32, device=dev)
        self.logits = torch.empty(self.B, cfg["vocab"], dtype=torch.float32, device=dev)
        ws = max(N.spd_prune_workspace_size(c) for c in self.cfgs)
        self.ws_prune = torch.zeros(ws, dtype=torch.uint8, device=dev)
        self.ws_proj = torch.zeros(N.spd_project_workspace_size(model, nv), dtype=torch.uint8, device=dev)
        self.ws_prefill = torch.zeros(N.spd_prefill_workspace_size(model, self.T, self.B), dtype=torch.uint8,
                                      device=dev)

    def run(self, feats, attn, text, skip_mask, stream=None):
        """feats[b]: list of [1][n_b][d_vis] fp32 per tapped layer, attn[b]: [1][H][n_b] received
        attention, text [sum(text_lens)][D] bf16. Returns the logits [B][vocab] (device)."""
        off = 0
        for b in range(self.B):
            k = self.keeps[b]
            if not self.dense:
                N.spd_prune(self.cfgs[b], feats[b], attn[b], self.keep_idx[b], ws=self.ws_prune, stream=stream)
            N.spd_gather_rows_bf16(feats[b][self.final_layer], 1, self.n_patches[b], self.d_vis, 0,
                                   self.keep_idx[b], k, self.vis[off:off + k], ws=self.ws_prune,
                                   stream=stream)
            off += k
        N.spd_project(self.model, self.vis, off, self.vis_rows, self.x, self.ws_proj, stream=stream)
        if len(self.text_rows):
            N.spd_scatter_rows(self.model, text, len(self.text_rows), self.text_rows, self.x, stream=stream)
        N.spd_prefill(self.model, self.x, self.T, self.cu, skip_mask, self.h, self.logits, self.ws_prefill,
                      stream=stream)
        return self.logits

    def status(self) -> int:
        codes = [N.spd_workspace_status(w) for w in (self.ws_prune, self.ws_proj, self.ws_prefill)]
        return next((c for c in codes if c), 0)
