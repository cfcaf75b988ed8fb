"""ctypes binding of libspider.so: the C ABI declared in include/spider.h, same names, argument
marshalling only (torch tensors -> device pointers, numpy arrays -> host pointers).

Importing this module loads nothing; the first call loads the in-tree library and raises if it
is missing. There is no fallback: every computation runs in the CUDA library.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "lib", "libspider.so")

SPD_OK, SPD_EINVAL, SPD_ENOSPC, SPD_ECUDA, SPD_ETIMEOUT, SPD_EUNSUPPORTED = 0, -1, -2, -3, -4, -5
SPD_MAX_FEAT_LAYERS = 4
EPI_F32, EPI_BF16, EPI_BIAS_BF16, EPI_BIAS_GELU_BF16, EPI_ADD_F32 = 0, 1, 2, 3, 4

# every symbol include/spider.h declares
EXPORTS = ("spd_last_error", "spd_workspace_status", "spd_selftest_bounded_wait",
           "spd_prune_workspace_size", "spd_prune_launches", "spd_prune", "spd_received_attention_workspace_size",
           "spd_received_attention", "spd_gather_rows_bf16", "spd_model_create",
           "spd_model_destroy", "spd_plan_adaptive", "spd_plan_static", "spd_project_workspace_size",
           "spd_project", "spd_scatter_rows", "spd_attention_workspace_size", "spd_attention",
           "spd_prefill_workspace_size", "spd_prefill", "spd_prefill_adaptive_workspace_size",
           "spd_prefill_adaptive", "spd_kv_cache_bytes", "spd_prefill_kv", "spd_decode_workspace_size",
           "spd_decode",
           "spd_linear_workspace_size", "spd_linear", "spd_linear_noalloc", "spd_trace_enable",
           "spd_trace_read", "spd_prune_workspace", "spd_prefill_workspace", "spd_gather_bf16",
           "spd_last_error_detail", "spd_check", "spd_plan_from_layer_mask", "spd_prefill_admit",
           "spd_stamp_enable", "spd_stamp_read", "spd_stamp_launch", "spd_set_deterministic",
           "spd_step_workspace_size", "spd_step", "spd_step_status")
TRACE_GEMM, TRACE_ATTN, TRACE_ROWS, TRACE_PRUNE = 0, 1, 2, 3


class SpiderError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"spider error {code}: {msg}")
        self.code = code


class PruneCfg(C.Structure):
    _fields_ = [("n_tiles", C.c_int), ("n_tok", C.c_int), ("has_cls", C.c_int), ("d_feat", C.c_int),
                ("n_layers", C.c_int), ("final_layer", C.c_int), ("n_heads", C.c_int),
                ("attn_form", C.c_int), ("keep", C.c_int), ("n_clusters", C.c_int),
                ("kmeans_iters", C.c_int), ("anchor_ratio", C.c_double),
                ("layer_weight", C.c_float * SPD_MAX_FEAT_LAYERS), ("sim_kind", C.c_int),
                ("ablate", C.c_int)]


SIM_KINDS = {"cos": 0, "mse": 1, "kl": 2}
SPD_PRUNE_NO_FINAL_SIM = 1
SPD_PRUNE_NO_ANCHOR_SIM = 2


class ModelCfg(C.Structure):
    _fields_ = [("n_layers", C.c_int), ("d_model", C.c_int), ("n_heads", C.c_int),
                ("n_kv_heads", C.c_int), ("head_dim", C.c_int), ("d_ffn", C.c_int),
                ("vocab", C.c_int), ("rope_theta", C.c_float), ("rms_eps", C.c_float),
                ("d_vis", C.c_int), ("d_proj", C.c_int)]


class SkipPolicy(C.Structure):
    _fields_ = [("t_skip", C.c_float), ("w1", C.c_float), ("w2", C.c_float), ("window", C.c_int),
                ("slc_norm", C.c_void_p), ("layer_target", C.c_void_p), ("is_visual", C.c_void_p),
                ("ablate", C.c_int), ("device_plan", C.c_int)]


SPD_SKIP_NO_ENTROPY = 1
SPD_SKIP_NO_ITC = 2
SPD_SKIP_NO_ACCUM = 4
SPD_SKIP_NO_SLC = 8


class LayerWeights(C.Structure):
    _fields_ = [(k, C.c_void_p) for k in ("attn_norm", "wq", "wk", "wv", "wo", "ffn_norm", "w_gate",
                                          "w_up", "w_down")]


class ModelWeights(C.Structure):
    _fields_ = [("layers", C.POINTER(LayerWeights))] + [
        (k, C.c_void_p) for k in ("final_norm", "lm_head", "proj_w1", "proj_b1", "proj_w2", "proj_b2")]


_lib = None


def lib():
    """The loaded library (loads it on first use; raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        vp, i, sz, ll = C.c_void_p, C.c_int, C.c_size_t, C.c_longlong
        sig = {
            "spd_last_error": (C.c_char_p, []),
            "spd_workspace_status": (i, [vp, vp, C.POINTER(i)]),
            "spd_selftest_bounded_wait": (i, [vp, ll, vp]),
            "spd_prune_workspace_size": (sz, [C.POINTER(PruneCfg)]),
            "spd_prune_launches": (i, [C.POINTER(PruneCfg)]),
            "spd_prune": (i, [C.POINTER(PruneCfg), C.POINTER(vp), vp, vp, vp, vp, vp, vp, sz, vp]),
            "spd_received_attention_workspace_size": (sz, [i, i, i]),
            "spd_received_attention": (i, [vp, i, i, i, vp, vp, i, vp, vp, sz, vp]),
            "spd_gather_rows_bf16": (i, [vp, i, i, i, i, vp, i, vp, vp, vp]),
            "spd_model_create": (i, [C.POINTER(ModelCfg), C.POINTER(ModelWeights), C.POINTER(vp)]),
            "spd_model_destroy": (None, [vp]),
            "spd_plan_adaptive": (i, [i, i, vp, vp, vp]),
            "spd_plan_static": (i, [i, i, vp, vp, vp]),
            "spd_project_workspace_size": (sz, [vp, i]),
            "spd_project": (i, [vp, vp, i, vp, vp, vp, sz, vp]),
            "spd_scatter_rows": (i, [vp, vp, i, vp, vp, vp]),
            "spd_attention_workspace_size": (sz, [i, i]),
            "spd_attention": (i, [vp, i, vp, vp, vp, i, vp, i, i, i, i, vp, vp, sz, vp]),
            "spd_prefill_workspace_size": (sz, [vp, i, i]),
            "spd_prefill": (i, [vp, vp, i, vp, i, vp, vp, vp, vp, sz, vp]),
            "spd_prune_workspace": (sz, [C.POINTER(PruneCfg)]),
            "spd_prefill_workspace": (sz, [vp, i, i]),
            "spd_gather_bf16": (i, [vp, i, vp, i, i, i, i, vp, vp]),
            "spd_last_error_detail": (i, [C.c_char_p, sz]),
            "spd_check": (i, [vp, vp]),
            "spd_plan_from_layer_mask": (i, [i, i, vp, vp, vp]),
            "spd_prefill_admit": (i, [vp, vp, i, vp, i, vp, vp, vp, vp, vp, sz, vp]),
            "spd_prefill_adaptive_workspace_size": (sz, [vp, i, i]),
            "spd_kv_cache_bytes": (sz, [vp, i, i]),
            "spd_prefill_kv": (i, [vp, vp, i, vp, i, vp, vp, vp, vp, i, vp, sz, vp]),
            "spd_decode_workspace_size": (sz, [vp, i]),
            "spd_decode": (i, [vp, vp, i, vp, vp, i, vp, vp, sz, vp]),
            "spd_prefill_adaptive": (i, [vp, vp, i, vp, i, C.POINTER(SkipPolicy), vp, vp, vp, vp, sz,
                                         vp]),
            "spd_linear_workspace_size": (sz, [i, i]),
            "spd_linear": (i, [vp, i, i, vp, i, i, vp, vp, vp, i, vp, sz, vp]),
            "spd_linear_noalloc": (i, [vp, i, i, vp, i, i, vp, vp, vp, i, vp, vp]),
            "spd_trace_enable": (i, [i]),
            "spd_set_deterministic": (i, [i]),
            "spd_step_workspace_size": (sz, [vp, C.POINTER(PruneCfg), i, vp, vp]),
            "spd_step": (i, [vp, C.POINTER(PruneCfg), i, vp, vp, C.POINTER(vp), vp, vp, vp, vp, vp, sz, vp]),
            "spd_step_status": (i, [vp, vp, C.POINTER(PruneCfg), i, vp, vp, vp]),
            "spd_stamp_enable": (i, [i]),
            "spd_stamp_launch": (i, [i, C.POINTER(i), C.POINTER(C.c_ulonglong), C.POINTER(C.c_ulonglong),
                                     C.POINTER(C.c_double), C.POINTER(C.c_double)]),
            "spd_stamp_read": (i, [i, C.POINTER(ll), C.POINTER(C.c_double), C.POINTER(C.c_double),
                                   C.POINTER(C.c_double)]),
            "spd_trace_read": (i, [i, C.POINTER(ll), C.POINTER(C.c_double), C.POINTER(C.c_double),
                                   C.POINTER(C.c_double)]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _check(rc: int):
    if rc != SPD_OK:
        raise SpiderError(rc, lib().spd_last_error().decode())


def _p(t):
    """Pointer for an argument: NULL for None, the host address of a numpy array (the wrappers
    below convert every host argument to one), the device address of a CUDA tensor. A tensor in
    host memory is refused: its address would reach a kernel as an invalid device pointer."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        if not t.flags["C_CONTIGUOUS"]:
            raise ValueError("host arrays passed to libspider must be C-contiguous")
        return t.ctypes.data
    if not getattr(t, "is_cuda", False):
        raise TypeError(f"device arguments of libspider must be CUDA tensors, got "
                        f"{type(t).__name__} on {getattr(t, 'device', 'the host')}")
    if not t.is_contiguous():
        raise ValueError("tensors passed to libspider must be contiguous")
    return t.data_ptr()


_DT = {"f32": "float32", "bf16": "bfloat16", "i32": "int32", "u8": "uint8", "i8": "int8"}


def _dev(t, dt, n, name, optional=False):
    """Device pointer of argument `name` after checking it: a contiguous CUDA tensor of element
    type dt ('f32', 'bf16', 'i32', 'u8', 'i8') holding at least n elements (the elements the call
    reads or writes). Raises before the library is called, so no kernel is handed a buffer that is
    too small, of the wrong type, or in host memory."""
    if t is None:
        if optional:
            return None
        raise ValueError(f"{name}: a device tensor is required")
    if isinstance(t, np.ndarray) or not getattr(t, "is_cuda", False):
        raise TypeError(f"{name}: device arguments of libspider must be CUDA tensors, got "
                        f"{type(t).__name__} on {getattr(t, 'device', 'the host')}")
    if str(t.dtype) != "torch." + _DT[dt]:
        raise ValueError(f"{name}: expected {_DT[dt]}, got {t.dtype}")
    if t.numel() < n:
        raise ValueError(f"{name}: {t.numel()} elements, the call touches {int(n)}")
    return _p(t)


def _host(a, dtype, n, name):
    """C-contiguous host copy of a host array argument with at least n elements."""
    a = np.ascontiguousarray(a, dtype=dtype)
    if a.size < n:
        raise ValueError(f"{name}: {a.size} elements, the call reads {int(n)}")
    return a


def _ws(ws):
    """Pointer and byte size of a workspace (a CUDA tensor of any element type)."""
    if ws is None:
        raise ValueError("ws: a device workspace is required")
    return _p(ws), ws.numel() * ws.element_size()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return int(stream)


def spd_last_error() -> str:
    return lib().spd_last_error().decode()


def spd_workspace_status(ws, stream=None) -> int:
    v = C.c_int(0)
    _check(lib().spd_workspace_status(_p(ws), _stream(stream), C.byref(v)))
    return v.value


def spd_selftest_bounded_wait(ws, budget_cycles: int, stream=None):
    _check(lib().spd_selftest_bounded_wait(_p(ws), int(budget_cycles), _stream(stream)))


def prune_cfg(n_tiles, n_tok, d_feat, n_layers, final_layer, n_heads, keep, *, has_cls=True,
              attn_form=0, n_clusters=4, kmeans_iters=10, anchor_ratio=0.7, layer_weight=None,
              sim="cos", use_final_sim=True, use_anchor_sim=True):
    w = list(layer_weight) if layer_weight is not None else [1.0] * SPD_MAX_FEAT_LAYERS
    w = w + [1.0] * (SPD_MAX_FEAT_LAYERS - len(w))
    ablate = (0 if use_final_sim else SPD_PRUNE_NO_FINAL_SIM) | (0 if use_anchor_sim else SPD_PRUNE_NO_ANCHOR_SIM)
    return PruneCfg(n_tiles, n_tok, int(has_cls), d_feat, n_layers, final_layer, n_heads, attn_form,
                    keep, n_clusters, kmeans_iters, float(anchor_ratio),
                    (C.c_float * SPD_MAX_FEAT_LAYERS)(*w), SIM_KINDS[sim], ablate)


def spd_prune_workspace_size(cfg: PruneCfg) -> int:
    return int(lib().spd_prune_workspace_size(C.byref(cfg)))


def spd_prune_launches(cfg: PruneCfg) -> int:
    """Kernels one spd_prune call with cfg enqueues on the current device."""
    n = int(lib().spd_prune_launches(C.byref(cfg)))
    _check(min(n, 0))
    return n


def spd_prune(cfg, feats, attn, keep_idx, kind=None, cluster=None, scores=None, ws=None, stream=None):
    T, n_tok, d = cfg.n_tiles, cfg.n_tok, cfg.d_feat
    n = n_tok - (1 if cfg.has_cls else 0)
    if len(feats) != cfg.n_layers:
        raise ValueError(f"feats: {len(feats)} layers, cfg.n_layers = {cfg.n_layers}")
    arr = (C.c_void_p * len(feats))(*[_dev(f, "f32", T * n_tok * d, f"feats[{i}]")
                                      for i, f in enumerate(feats)])
    n_att = n_tok if cfg.attn_form == 0 else n
    wp, wb = _ws(ws)
    _check(lib().spd_prune(C.byref(cfg), arr, _dev(attn, "f32", T * cfg.n_heads * n_att, "attn"),
                           _dev(keep_idx, "i32", T * cfg.keep, "keep_idx"),
                           _dev(kind, "u8", T * n, "kind", True), _dev(cluster, "i8", T * n, "cluster", True),
                           _dev(scores, "f32", T * n, "scores", True), wp, wb, _stream(stream)))


def spd_received_attention_workspace_size(n_maps: int, n_q: int, n_k: int) -> int:
    return int(lib().spd_received_attention_workspace_size(n_maps, n_q, n_k))


def spd_received_attention(maps, out, ws, group_start=None, group_members=None, stream=None):
    """Received-attention form out [n_maps][n_out] from full maps [n_maps][n_q][n_k] (optionally
    through a patch merger given as CSR groups)."""
    n_maps, n_q, n_k = maps.shape
    n_out = out.shape[-1]
    if (group_start is None) != (group_members is None):
        raise ValueError("group_start and group_members go together")
    wp, wb = _ws(ws)
    _check(lib().spd_received_attention(_dev(maps, "f32", n_maps * n_q * n_k, "maps"), n_maps, n_q, n_k,
                                        _dev(group_start, "i32", n_out + 1, "group_start", True),
                                        _dev(group_members, "i32", 1, "group_members", True),
                                        n_out, _dev(out, "f32", n_maps * n_out, "out"), wp, wb,
                                        _stream(stream)))


def spd_gather_rows_bf16(src, n_tiles, n_tok, d, row_offset, idx, keep, dst, ws=None, stream=None):
    _check(lib().spd_gather_rows_bf16(_dev(src, "f32", n_tiles * n_tok * d, "src"), n_tiles, n_tok, d,
                                      row_offset, _dev(idx, "i32", n_tiles * keep, "idx"), keep,
                                      _dev(dst, "bf16", n_tiles * keep * d, "dst"), _p(ws),
                                      _stream(stream)))


class SpdModel:
    """Owner of an spd_model handle (spd_model_create / spd_model_destroy)."""

    def __init__(self, cfg: dict, weights: dict):
        self.cfg = dict(cfg)
        mc = ModelCfg(cfg["n_layers"], cfg["d_model"], cfg["n_heads"], cfg["n_kv_heads"],
                      cfg["head_dim"], cfg["d_ffn"], cfg["vocab"], float(cfg["rope_theta"]),
                      float(cfg["rms_eps"]), cfg.get("d_vis", 0) if cfg.get("d_proj") else 0,
                      cfg.get("d_proj", 0))
        D, H, Hkv, hd, F = (cfg[k] for k in ("d_model", "n_heads", "n_kv_heads", "head_dim", "d_ffn"))
        shapes = dict(attn_norm=D, wq=H * hd * D, wk=Hkv * hd * D, wv=Hkv * hd * D, wo=D * H * hd,
                      ffn_norm=D, w_gate=F * D, w_up=F * D, w_down=D * F)
        if len(weights["layers"]) != cfg["n_layers"]:
            raise ValueError(f"weights: {len(weights['layers'])} layers, n_layers = {cfg['n_layers']}")
        layers = (LayerWeights * cfg["n_layers"])()
        for l, lw in enumerate(weights["layers"]):
            for k, _ in LayerWeights._fields_:
                setattr(layers[l], k, _dev(lw[k], "bf16", shapes[k], f"layers[{l}].{k}"))
        dv, dp = mc.d_vis, mc.d_proj
        proj = [_dev(weights.get(k), "bf16", n, k, optional=not dp)
                for k, n in (("proj_w1", dp * dv), ("proj_b1", dp), ("proj_w2", D * dp), ("proj_b2", D))]
        mw = ModelWeights(layers, _dev(weights["final_norm"], "bf16", D, "final_norm"),
                          _dev(weights["lm_head"], "bf16", cfg["vocab"] * D, "lm_head"), *proj)
        h = C.c_void_p()
        import torch
        torch.cuda.synchronize()
        _check(lib().spd_model_create(C.byref(mc), C.byref(mw), C.byref(h)))
        self.handle = h

    def close(self):
        if getattr(self, "handle", None):
            lib().spd_model_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def spd_plan_adaptive(n_layers: int, admit: np.ndarray, target: np.ndarray) -> np.ndarray:
    admit = np.ascontiguousarray(admit, dtype=np.int16)
    target = _host(target, np.uint8, len(admit), "target")
    mask = np.zeros((n_layers, len(admit)), dtype=np.uint8)
    _check(lib().spd_plan_adaptive(n_layers, len(admit), _p(admit), _p(target), _p(mask)))
    return mask


def spd_plan_static(layer_mask: np.ndarray, token_sel: np.ndarray) -> np.ndarray:
    layer_mask = np.ascontiguousarray(layer_mask, dtype=np.uint8)
    token_sel = np.ascontiguousarray(token_sel, dtype=np.uint8)
    mask = np.zeros((len(layer_mask), len(token_sel)), dtype=np.uint8)
    _check(lib().spd_plan_static(len(layer_mask), len(token_sel), _p(layer_mask), _p(token_sel),
                                 _p(mask)))
    return mask


def spd_project_workspace_size(model: SpdModel, rows: int) -> int:
    return int(lib().spd_project_workspace_size(model.handle, rows))


def spd_project(model: SpdModel, vis, rows, out_rows, x, ws, stream=None):
    """Projector of `rows` bf16 vision rows into rows out_rows[i] of x (row indices must lie inside
    x: device values, not read back here)."""
    D = model.cfg["d_model"]
    wp, wb = _ws(ws)
    _check(lib().spd_project(model.handle, _dev(vis, "bf16", rows * model.cfg.get("d_vis", 0), "vis"),
                             rows, _dev(out_rows, "i32", rows, "out_rows"),
                             _dev(x, "bf16", min(rows, 1) * D, "x"), wp, wb, _stream(stream)))


def spd_attention_workspace_size(n_q: int, n_seqs: int) -> int:
    return int(lib().spd_attention_workspace_size(n_q, n_seqs))


def spd_attention(q, q_pos, q_cu, kv, cu_seqlens, n_heads, n_kv_heads, head_dim, o, ws, stream=None):
    """Causal attention of the query rows q (positions q_pos, sequences delimited by the host
    array q_cu) over the K/V rows kv of their sequences (host cu_seqlens); writes o."""
    q_cu = np.ascontiguousarray(q_cu, dtype=np.int32)
    cu = _host(cu_seqlens, np.int32, len(q_cu), "cu_seqlens")
    n_q, n_kv = int(q_cu[-1]), int(cu[-1])
    qd, kvd = n_heads * head_dim, n_kv_heads * head_dim
    wp, wb = _ws(ws)
    _check(lib().spd_attention(_dev(q, "bf16", n_q * qd, "q"), n_q, _dev(q_pos, "i32", n_q, "q_pos"),
                               _p(q_cu), _dev(kv, "bf16", n_kv * 2 * kvd, "kv"), n_kv, _p(cu),
                               len(q_cu) - 1, n_heads, n_kv_heads, head_dim,
                               _dev(o, "bf16", n_q * qd, "o"), wp, wb, _stream(stream)))


def spd_scatter_rows(model: SpdModel, src, rows, rows_map, dst, stream=None):
    """dst[rows_map[i]] = src[i] for `rows` bf16 rows of d_model (row indices must lie inside dst:
    device values, not read back here)."""
    D = model.cfg["d_model"]
    _check(lib().spd_scatter_rows(model.handle, _dev(src, "bf16", rows * D, "src"), rows,
                                  _dev(rows_map, "i32", rows, "rows_map"),
                                  _dev(dst, "bf16", min(rows, 1) * D, "dst"), _stream(stream)))


def spd_prefill_workspace_size(model: SpdModel, max_tokens: int, max_seqs: int) -> int:
    return int(lib().spd_prefill_workspace_size(model.handle, max_tokens, max_seqs))


def spd_prefill_adaptive_workspace_size(model: SpdModel, max_tokens: int, max_seqs: int) -> int:
    return int(lib().spd_prefill_adaptive_workspace_size(model.handle, max_tokens, max_seqs))


def spd_prefill_adaptive(model: SpdModel, x, n_tokens, cu_seqlens, is_visual, slc_norm, layer_target,
                         t_skip, w1, w2, window, h, logits, ws, stream=None, ablate=0, device_plan=0):
    """Prefill with the online ASL-Skip plan; returns the admission layer of every token (host
    int16, -1 = never). ablate: bit set of SPD_SKIP_NO_*; device_plan: decisions and row lists on
    the device (1) or read back per window layer (0)."""
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    L, D, B = model.cfg["n_layers"], model.cfg["d_model"], len(cu) - 1
    slc = _host(slc_norm, np.float32, L, "slc_norm")
    tgt = _host(layer_target, np.uint8, L, "layer_target")
    vis = _host(is_visual, np.uint8, n_tokens, "is_visual")
    admit = np.full(n_tokens, -9, dtype=np.int16)
    pol = SkipPolicy(float(t_skip), float(w1), float(w2), int(window), slc.ctypes.data, tgt.ctypes.data,
                     vis.ctypes.data, int(ablate), int(device_plan))
    wp, wb = _ws(ws)
    _check(lib().spd_prefill_adaptive(model.handle, _dev(x, "bf16", n_tokens * D, "x"), n_tokens,
                                      cu.ctypes.data, B, C.byref(pol), admit.ctypes.data,
                                      _dev(h, "f32", n_tokens * D, "h"),
                                      _dev(logits, "f32", B * model.cfg["vocab"], "logits", True), wp, wb,
                                      _stream(stream)))
    return admit


def spd_kv_cache_bytes(model: SpdModel, n_seqs: int, max_len: int) -> int:
    return int(lib().spd_kv_cache_bytes(model.handle, n_seqs, max_len))


def spd_prefill_kv(model: SpdModel, x, n_tokens, cu_seqlens, skip_mask, h, logits, kv_cache, max_len, ws,
                   stream=None):
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    L, D, B = model.cfg["n_layers"], model.cfg["d_model"], len(cu) - 1
    mk = None if skip_mask is None else _host(skip_mask, np.uint8, L * n_tokens, "skip_mask")
    wp, wb = _ws(ws)
    _check(lib().spd_prefill_kv(model.handle, _dev(x, "bf16", n_tokens * D, "x"), n_tokens, cu.ctypes.data,
                                B, None if mk is None else mk.ctypes.data, _dev(h, "f32", n_tokens * D, "h"),
                                _dev(logits, "f32", B * model.cfg["vocab"], "logits", True),
                                _dev(kv_cache, "bf16", spd_kv_cache_bytes(model, B, max_len) // 2, "kv_cache"),
                                max_len, wp, wb, _stream(stream)))


def spd_decode_workspace_size(model: SpdModel, n_seqs: int) -> int:
    return int(lib().spd_decode_workspace_size(model.handle, n_seqs))


def spd_decode(model: SpdModel, x, pos, kv_cache, max_len, logits, ws, stream=None):
    p = np.ascontiguousarray(pos, dtype=np.int32)
    B, D = len(p), model.cfg["d_model"]
    wp, wb = _ws(ws)
    _check(lib().spd_decode(model.handle, _dev(x, "bf16", B * D, "x"), B, p.ctypes.data,
                            _dev(kv_cache, "bf16", spd_kv_cache_bytes(model, B, max_len) // 2, "kv_cache"),
                            max_len, _dev(logits, "f32", B * model.cfg["vocab"], "logits"), wp, wb,
                            _stream(stream)))


def spd_prefill(model: SpdModel, x, n_tokens, cu_seqlens, skip_mask, h, logits, ws, stream=None):
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    L, D, B = model.cfg["n_layers"], model.cfg["d_model"], len(cu) - 1
    mask = None if skip_mask is None else _host(skip_mask, np.uint8, L * n_tokens, "skip_mask")
    wp, wb = _ws(ws)
    _check(lib().spd_prefill(model.handle, _dev(x, "bf16", n_tokens * D, "x"), n_tokens, _p(cu), B,
                             _p(mask), _dev(h, "f32", n_tokens * D, "h"),
                             _dev(logits, "f32", B * model.cfg["vocab"], "logits", True), wp, wb,
                             _stream(stream)))


def spd_prefill_admit(model: SpdModel, x, n_tokens, cu_seqlens, admit_layer, target, h, logits, ws,
                      stream=None):
    """spd_prefill with the per-token plan (admission layer, frozen target), expanded on the host."""
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    D, B = model.cfg["d_model"], len(cu) - 1
    ad = None if admit_layer is None else _host(admit_layer, np.int16, n_tokens, "admit_layer")
    tg = None if target is None else _host(target, np.uint8, n_tokens, "target")
    wp, wb = _ws(ws)
    _check(lib().spd_prefill_admit(model.handle, _dev(x, "bf16", n_tokens * D, "x"), n_tokens, _p(cu), B,
                                   _p(ad), _p(tg), _dev(h, "f32", n_tokens * D, "h"),
                                   _dev(logits, "f32", B * model.cfg["vocab"], "logits", True), wp, wb,
                                   _stream(stream)))


def spd_check(ws, stream=None) -> int:
    """Device-side status of a workspace (reads and clears it; synchronises the stream)."""
    return int(lib().spd_check(_p(ws), _stream(stream)))


def spd_last_error_detail() -> str:
    buf = C.create_string_buffer(512)
    lib().spd_last_error_detail(buf, 512)
    return buf.value.decode()


def spd_linear_workspace_size(M: int, N: int) -> int:
    return int(lib().spd_linear_workspace_size(M, N))


def _linear_args(X, M, K, W, N, epilogue, out, ldo, bias, rows):
    """Checked pointers of a linear call: out holds M rows of ldo (or, with a row map, at least one
    row: the map's device values must lie inside out and are not read back here)."""
    out_dt = "f32" if epilogue in (EPI_F32, EPI_ADD_F32) else "bf16"
    out_n = (ldo if rows is not None else M * ldo) if M > 0 else 0
    return (_dev(X, "bf16", M * K, "X"), _dev(W, "bf16", N * K, "W"),
            _dev(bias, "bf16", N, "bias", True), _dev(rows, "i32", M, "rows", True),
            _dev(out, out_dt, out_n, "out"))


def spd_linear(X, M, K, W, N, epilogue, out, ldo, ws, bias=None, rows=None, stream=None):
    x, w, b, r, o = _linear_args(X, M, K, W, N, epilogue, out, ldo, bias, rows)
    wp, wb = _ws(ws)
    _check(lib().spd_linear(x, M, K, w, N, epilogue, b, r, o, ldo, wp, wb, _stream(stream)))


def spd_linear_noalloc(X, M, K, W, N, epilogue, out, ldo, bias=None, rows=None, status=None,
                       stream=None):
    """spd_linear with the library's own static scratch instead of a caller workspace."""
    x, w, b, r, o = _linear_args(X, M, K, W, N, epilogue, out, ldo, bias, rows)
    _check(lib().spd_linear_noalloc(x, M, K, w, N, epilogue, b, r, o, ldo,
                                    _dev(status, "i32", 1, "status", True), _stream(stream)))


def spd_trace_enable(capacity: int):
    _check(lib().spd_trace_enable(int(capacity)))


def spd_trace_read(cls: int) -> dict:
    """Launch count, device ms, algorithmic flops and bytes of one kernel class (synchronises)."""
    n, ms, fl, by = C.c_longlong(), C.c_double(), C.c_double(), C.c_double()
    _check(lib().spd_trace_read(cls, C.byref(n), C.byref(ms), C.byref(fl), C.byref(by)))
    return dict(launches=n.value, ms=ms.value, flops=fl.value, bytes=by.value)


def spd_stamp_enable(capacity: int):
    _check(lib().spd_stamp_enable(int(capacity)))


def spd_stamp_read(cls: int) -> dict:
    """Launch count, stamped device ms, algorithmic flops and bytes of one kernel class (device
    globaltimer stamps; synchronises)."""
    n, ms, fl, by = C.c_longlong(), C.c_double(), C.c_double(), C.c_double()
    _check(lib().spd_stamp_read(cls, C.byref(n), C.byref(ms), C.byref(fl), C.byref(by)))
    return dict(launches=n.value, ms=ms.value, flops=fl.value, bytes=by.value)


def spd_stamp_launches() -> list:
    """Every stamped launch since spd_stamp_enable, in launch order: (class, start ns, end ns,
    flops, bytes)."""
    out = []
    k = 0
    cls, s0, s1 = C.c_int(), C.c_ulonglong(), C.c_ulonglong()
    fl, by = C.c_double(), C.c_double()
    while lib().spd_stamp_launch(k, C.byref(cls), C.byref(s0), C.byref(s1), C.byref(fl), C.byref(by)) == SPD_OK:
        out.append((cls.value, s0.value, s1.value, fl.value, by.value))
        k += 1
    return out


def spd_set_deterministic(on: bool):
    """Library-wide deterministic mode: GEMM sums in a fixed order (bit-identical repeated runs)."""
    _check(lib().spd_set_deterministic(int(bool(on))))


def _any(t, dt, n, name, optional=False):
    """Pointer of an argument that may be in host or device memory (spd_step): a contiguous torch
    tensor of element type dt with at least n elements, on the GPU or the CPU (pinned or not)."""
    if t is None:
        if optional:
            return None
        raise ValueError(f"{name}: a tensor is required")
    if getattr(t, "is_cuda", False):
        return _dev(t, dt, n, name)
    if isinstance(t, np.ndarray) or not hasattr(t, "data_ptr"):
        raise TypeError(f"{name}: a torch tensor is required")
    if str(t.dtype) != "torch." + _DT[dt]:
        raise ValueError(f"{name}: expected {_DT[dt]}, got {t.dtype}")
    if t.numel() < n:
        raise ValueError(f"{name}: {t.numel()} elements, the call touches {int(n)}")
    if not t.is_contiguous():
        raise ValueError(f"{name}: must be contiguous")
    return t.data_ptr()


def _step_layout(cfg, tiles_per_seq, text_len):
    tps = np.ascontiguousarray(tiles_per_seq, dtype=np.int32)
    tl = _host(text_len, np.int32, len(tps), "text_len")
    return tps, tl


def spd_step_workspace_size(model: SpdModel, cfg, tiles_per_seq, text_len) -> int:
    tps, tl = _step_layout(cfg, tiles_per_seq, text_len)
    return int(lib().spd_step_workspace_size(model.handle, C.byref(cfg), len(tps), tps.ctypes.data,
                                             tl.ctypes.data))


def spd_step(model: SpdModel, cfg, tiles_per_seq, text_len, feats, attn, text, skip_mask, logits, ws,
             stream=None):
    """The whole SPIDER step (prune, gather, projector, text rows, prefill) in one call; feats,
    attn, text and logits may be host (CPU) or device tensors."""
    tps, tl = _step_layout(cfg, tiles_per_seq, text_len)
    B, D, L = len(tps), model.cfg["d_model"], model.cfg["n_layers"]
    T = int(tps.sum()) * cfg.keep + int(tl.sum())
    n = cfg.n_tok - (1 if cfg.has_cls else 0)
    n_att = cfg.n_tok if cfg.attn_form == 0 else n
    if len(feats) != cfg.n_layers:
        raise ValueError(f"feats: {len(feats)} layers, cfg.n_layers = {cfg.n_layers}")
    fa = (C.c_void_p * len(feats))(*[_any(f, "f32", cfg.n_tiles * cfg.n_tok * cfg.d_feat, f"feats[{i}]")
                                      for i, f in enumerate(feats)])
    mask = None if skip_mask is None else _host(skip_mask, np.uint8, L * T, "skip_mask")
    wp, wb = _ws(ws)
    _check(lib().spd_step(model.handle, C.byref(cfg), B, tps.ctypes.data, tl.ctypes.data, fa,
                          _any(attn, "f32", cfg.n_tiles * cfg.n_heads * n_att, "attn"),
                          _any(text, "bf16", int(tl.sum()) * D, "text", optional=int(tl.sum()) == 0),
                          None if mask is None else mask.ctypes.data,
                          _any(logits, "f32", B * model.cfg["vocab"], "logits"), wp, wb, _stream(stream)))


def spd_step_status(ws, model: SpdModel, cfg, tiles_per_seq, text_len, stream=None) -> int:
    tps, tl = _step_layout(cfg, tiles_per_seq, text_len)
    return int(lib().spd_step_status(_p(ws), model.handle, C.byref(cfg), len(tps), tps.ctypes.data,
                                     tl.ctypes.data, _stream(stream)))
