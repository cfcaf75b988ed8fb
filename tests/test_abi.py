"""Host-side checks of libspider.so (no GPU needed): the library loads, exports every entry point
include/spider.h declares, and its host-only logic (plan expansion, argument validation) matches
the oracle."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from oracle import decoder as od
from paper_2609_34977_gb300 import _native as N

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(N.LIB_PATH):
        from paper_2609_34977_gb300 import build
        build.build()
    return N.lib()


def declared_functions():
    src = open(os.path.join(ROOT, "include", "spider.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(spd_\w+)\s*\(", src)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(N.EXPORTS)


@pytest.mark.parametrize("seed", range(5))
def test_adaptive_plan_matches_oracle(lib, seed):
    r = np.random.default_rng(seed)
    T, L = 50, 7
    admit = r.integers(-1, L, size=T).astype(np.int16)
    target = r.integers(1, 3, size=T).astype(np.uint8)
    np.testing.assert_array_equal(N.spd_plan_adaptive(L, admit, target),
                                  od.expand_adaptive_plan(admit, target, L))


def test_static_plan_matches_oracle(lib):
    lm = np.array([0, 2, 1, 3], dtype=np.uint8)
    sel = np.array([1, 0, 1, 1, 0], dtype=np.uint8)
    np.testing.assert_array_equal(N.spd_plan_static(lm, sel), od.expand_static_plan(lm, sel))


def test_plan_rejects_bad_target(lib):
    with pytest.raises(N.SpiderError) as e:
        N.spd_plan_adaptive(3, np.array([0], np.int16), np.array([5], np.uint8))
    assert e.value.code == N.SPD_EINVAL


def test_prune_config_validation(lib):
    good = N.prune_cfg(1, 577, 256, 3, 2, 8, 64)
    assert N.spd_prune_workspace_size(good) > 0
    for bad in (N.prune_cfg(1, 577, 256, 3, 3, 8, 64),      # final layer out of range
                N.prune_cfg(1, 577, 250, 3, 2, 8, 64),      # d not a multiple of 4
                N.prune_cfg(1, 577, 256, 3, 2, 8, 577),     # keep > n_patch
                N.prune_cfg(1, 577, 256, 3, 2, 8, 64, n_clusters=17),
                N.prune_cfg(1, 577, 256, 3, 2, 8, 64, anchor_ratio=1.5),
                N.prune_cfg(1, 576, 256, 3, 2, 8, 64, has_cls=False, attn_form=0)):
        assert N.spd_prune_workspace_size(bad) == 0


def test_workspace_sizes_grow_with_problem(lib):
    a = N.spd_prune_workspace_size(N.prune_cfg(1, 577, 1024, 2, 1, 16, 192))
    b = N.spd_prune_workspace_size(N.prune_cfg(5, 577, 1024, 2, 1, 16, 64))
    assert b > a > 0
    assert N.spd_linear_workspace_size(256, 4096) > 0


def test_contract_names_are_the_same_calls(lib):
    cfg = N.prune_cfg(2, 577, 64, 2, 1, 4, 32)
    assert lib.spd_prune_workspace(C.byref(cfg)) == lib.spd_prune_workspace_size(C.byref(cfg)) > 0
    lm = np.array([0, 2, 1], dtype=np.uint8)
    sel = np.array([1, 0, 1, 1], dtype=np.uint8)
    a = np.zeros(12, np.uint8)
    b = np.zeros(12, np.uint8)
    assert lib.spd_plan_from_layer_mask(3, 4, lm.ctypes.data, sel.ctypes.data, a.ctypes.data) == 0
    assert lib.spd_plan_static(3, 4, lm.ctypes.data, sel.ctypes.data, b.ctypes.data) == 0
    np.testing.assert_array_equal(a, b)
    # a rejected call's message through both forms; truncation to the buffer
    with pytest.raises(N.SpiderError):
        N.spd_plan_adaptive(3, np.array([0], np.int16), np.array([5], np.uint8))
    assert N.spd_last_error_detail() == N.lib().spd_last_error().decode()
    small = C.create_string_buffer(5)
    n = lib.spd_last_error_detail(small, 5)
    assert n == len(N.lib().spd_last_error()) and len(small.value) == 4


def test_plan_accepts_both_sublayers_target(lib):
    mask = N.spd_plan_adaptive(3, np.array([1, -1], np.int16), np.array([3, 1], np.uint8))
    np.testing.assert_array_equal(mask, [[0, 0], [3, 0], [3, 0]])


def test_missing_library_raises_instead_of_falling_back(monkeypatch, tmp_path):
    # the product path has no CPU fallback: without the built library every call raises
    monkeypatch.setattr(N, "_lib", None)
    monkeypatch.setattr(N, "LIB_PATH", str(tmp_path / "libspider.so"))
    with pytest.raises(RuntimeError, match="is missing"):
        N.lib()
    with pytest.raises(RuntimeError, match="is missing"):
        N.spd_plan_adaptive(2, np.array([0, -1], np.int16), np.array([1, 0], np.uint8))


def test_plan_expansions_match_oracle_over_random_shapes(lib):
    # per-token (admission layer, target in 1..3) and per-layer masks, 1..40 layers, 1..300 tokens
    r = np.random.default_rng(77)
    for _ in range(60):
        L, T = int(r.integers(1, 41)), int(r.integers(1, 301))
        admit = r.integers(-1, L, size=T).astype(np.int16)
        target = r.integers(1, 4, size=T).astype(np.uint8)
        np.testing.assert_array_equal(N.spd_plan_adaptive(L, admit, target),
                                      od.expand_adaptive_plan(admit, target, L))
        lm = r.integers(0, 4, size=L).astype(np.uint8)
        sel = (r.random(T) < 0.6).astype(np.uint8)
        np.testing.assert_array_equal(N.spd_plan_static(lm, sel), od.expand_static_plan(lm, sel))


def test_plan_admission_edges(lib):
    # an admission at or past the last layer never takes effect; a token never admitted may carry
    # any target; an admitted token's target must name a sub-layer
    mask = N.spd_plan_adaptive(3, np.array([3, -1, -5, 2], np.int16), np.array([1, 0, 9, 2], np.uint8))
    np.testing.assert_array_equal(mask, [[0, 0, 0, 0], [0, 0, 0, 0], [0, 0, 0, 2]])
    with pytest.raises(N.SpiderError) as e:
        N.spd_plan_adaptive(3, np.array([0], np.int16), np.array([0], np.uint8))
    assert e.value.code == N.SPD_EINVAL


def test_host_tensor_for_a_device_argument_is_refused(lib):
    # refused in the binding, before the library is called: no kernel sees a host address
    import torch
    with pytest.raises(TypeError, match="CUDA tensors"):
        N.spd_workspace_status(torch.zeros(16, dtype=torch.uint8))


class _FakeCuda:
    """Stands in for a CUDA tensor in the binding's argument checks (no GPU here): the checks must
    refuse it before the library is called, so its pointer is never used."""

    def __init__(self, dtype, numel):
        import torch
        self.dtype = getattr(torch, dtype)
        self.is_cuda = True
        self._n = numel

    def numel(self):
        return self._n

    def element_size(self):
        return 1

    def is_contiguous(self):
        return True

    def data_ptr(self):
        return 0


def test_binding_refuses_undersized_or_mistyped_device_arguments(lib):
    M, K, Nw = 64, 256, 128
    ok = dict(X=_FakeCuda("bfloat16", M * K), W=_FakeCuda("bfloat16", Nw * K),
              out=_FakeCuda("float32", M * Nw))
    bad = [dict(X=_FakeCuda("bfloat16", M * K - 1)),            # X one element short
           dict(W=_FakeCuda("float32", Nw * K)),                 # fp32 weights where bf16 is read
           dict(out=_FakeCuda("float32", M * Nw - 8)),           # output rows past the end
           dict(out=_FakeCuda("bfloat16", M * Nw)),              # bf16 output for an fp32 epilogue
           dict(X=np.zeros((M, K), np.float32))]                 # a host array for a device pointer
    for b in bad:
        a = dict(ok, **b)
        with pytest.raises((ValueError, TypeError)):
            N.spd_linear(a["X"], M, K, a["W"], Nw, N.EPI_F32, a["out"], Nw, _FakeCuda("uint8", 1 << 30))
        with pytest.raises((ValueError, TypeError)):
            N.spd_linear_noalloc(a["X"], M, K, a["W"], Nw, N.EPI_F32, a["out"], Nw)
    with pytest.raises(ValueError):  # a residual status word of the wrong type
        N.spd_linear_noalloc(ok["X"], M, K, ok["W"], Nw, N.EPI_F32, ok["out"], Nw,
                             status=_FakeCuda("float32", 1))


def test_binding_refuses_short_host_arrays_and_buffers_of_prune_and_gather(lib):
    cfg = N.prune_cfg(2, 577, 64, 2, 1, 4, 32)
    feats = [_FakeCuda("float32", 2 * 577 * 64)] * 2
    attn = _FakeCuda("float32", 2 * 4 * 577)
    idx = _FakeCuda("int32", 2 * 32)
    ws = _FakeCuda("uint8", 1 << 20)
    for kw in (dict(feats=[feats[0]]),                                  # one layer missing
               dict(attn=_FakeCuda("float32", 2 * 4 * 576)),            # the CLS rows are 577 wide
               dict(idx=_FakeCuda("int32", 63)),
               dict(kind=_FakeCuda("uint8", 2 * 576 - 1))):
        a = dict(feats=feats, attn=attn, idx=idx, kind=None) | kw
        with pytest.raises(ValueError):
            N.spd_prune(cfg, a["feats"], a["attn"], a["idx"], kind=a["kind"], ws=ws)
    with pytest.raises(ValueError):
        N.spd_gather_rows_bf16(feats[0], 2, 577, 64, 1, idx, 32, _FakeCuda("bfloat16", 2 * 32 * 64 - 1))


def test_binding_refuses_short_plans_and_residual_buffers(lib):
    class M:  # a model handle is never reached: the checks come first
        cfg = dict(n_layers=3, d_model=64, vocab=10)
        handle = None
    T = 20
    x, h = _FakeCuda("bfloat16", T * 64), _FakeCuda("float32", T * 64)
    ws = _FakeCuda("uint8", 1 << 20)
    with pytest.raises(ValueError):  # skip mask of 2 layers for a 3-layer model
        N.spd_prefill(M, x, T, [0, T], np.zeros((2, T), np.uint8), h, None, ws)
    with pytest.raises(ValueError):  # residual stream one row short
        N.spd_prefill(M, x, T, [0, T], None, _FakeCuda("float32", (T - 1) * 64), None, ws)
    with pytest.raises(ValueError):  # logits of one sequence for two
        N.spd_prefill(M, x, T, [0, 5, T], None, h, _FakeCuda("float32", 10), ws)
    with pytest.raises(ValueError):  # per-token plan shorter than the tokens
        N.spd_prefill_admit(M, x, T, [0, T], np.zeros(T - 1, np.int16), np.ones(T, np.uint8), h, None, ws)
