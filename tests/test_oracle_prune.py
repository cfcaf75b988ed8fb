"""Pins of the MSV-Prune oracle (§4.1, Eq. 1-3) against brute force, closed forms and invariants.

None of these re-types the oracle's own formula: each check computes the expected result another
way (exhaustive search, a mathematically equivalent identity, textbook special cases).
"""
import itertools
import json
import os

import numpy as np
import pytest

from oracle import prune as op
from paper_2609_34977_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_attention_importance_drops_cls_column_and_averages_heads():
    a = np.zeros((3, 5))
    a[:, 0] = 100.0                     # CLS -> CLS, must not count
    a[0, 1:] = [1, 2, 3, 4]
    a[1, 1:] = [3, 2, 1, 0]
    a[2, 1:] = [2, 2, 2, 2]
    np.testing.assert_array_equal(op.attention_importance(a, 0), [2.0, 2.0, 2.0, 2.0])
    np.testing.assert_array_equal(op.attention_importance(a[:, 1:], 1), [2.0, 2.0, 2.0, 2.0])


@pytest.mark.parametrize("seed", range(6))
def test_anchor_topk_equals_exhaustive_search(seed):
    r = np.random.default_rng(seed)
    n = 9
    a = r.integers(0, 4, size=n).astype(float)     # many ties on purpose
    for k in range(n + 1):
        best = None
        for sub in itertools.combinations(range(n), k):   # sorted tuples
            key = (-sum(a[list(sub)]), sub)                 # max sum, then lowest indices
            if best is None or key < best[0]:
                best = (key, sub)
        assert tuple(op.select_anchors(a, k)) == best[1]


def test_n_anchor_rounding():
    assert op.n_anchor_tokens(192, 0.7) == 134
    assert op.n_anchor_tokens(128, 0.7) == 90
    assert op.n_anchor_tokens(64, 0.7) == 45
    assert op.n_anchor_tokens(10, 0.25) == 3     # 2.5 rounds away from zero
    assert op.n_anchor_tokens(64, 0.0) == 0
    assert op.n_anchor_tokens(64, 1.0) == 64


def test_quota_golden_cases():
    with open(os.path.join(GOLDEN, "eq2_quotas.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        assert op.cluster_quotas(c["sizes"], c["n_cmp"]) == c["quota"], c["why"]


@pytest.mark.parametrize("seed", range(20))
def test_quota_invariants(seed):
    r = np.random.default_rng(seed)
    sizes = r.integers(0, 30, size=int(r.integers(1, 8))).tolist()
    total = sum(sizes)
    n_cmp = int(r.integers(0, total + 1)) if total else 0
    q = op.cluster_quotas(sizes, n_cmp)
    assert sum(q) == n_cmp
    assert all(0 <= qk <= sk for qk, sk in zip(q, sizes))
    nonempty = sum(1 for s in sizes if s)
    if n_cmp >= nonempty:
        assert all(qk >= 1 for qk, sk in zip(q, sizes) if sk)   # Eq. 2's floor of one


def _planted(r, n, d, k, sep=10.0, noise=1.0):
    z = (np.arange(n) * k) // n
    mu = sep * r.standard_normal((k, d))
    return mu[z] + noise * r.standard_normal((n, d)), z


def test_kmeans_recovers_planted_bands():
    r = np.random.default_rng(1)
    x, z = _planted(r, 60, 8, 3)
    assign, margin = op.kmeans(x, 3, 10)
    np.testing.assert_array_equal(assign, z)
    assert margin > 1.0


@pytest.mark.parametrize("seed", range(4))
def test_kmeans_matches_exhaustive_min_sse(seed):
    r = np.random.default_rng(100 + seed)
    n = 11
    x, _ = _planted(r, n, 3, 2, sep=6.0)
    best = None
    for bits in range(1, 2 ** (n - 1)):       # every 2-way partition (label 0 holds point 0)
        lab = np.array([(bits >> i) & 1 for i in range(n)])
        if lab.sum() == 0:
            continue
        sse = sum(((x[lab == c] - x[lab == c].mean(0)) ** 2).sum() for c in (0, 1))
        if best is None or sse < best[0]:
            best = (sse, lab)
    assign, _ = op.kmeans(x, 2, 50)
    same = np.array_equal(assign, best[1]) or np.array_equal(assign, 1 - best[1])
    assert same


def test_kmeans_converged_assignment_is_a_fixed_point():
    r = np.random.default_rng(7)
    x = r.standard_normal((80, 5))
    assign, _ = op.kmeans(x, 4, 200)
    c = np.stack([x[assign == k].mean(0) for k in range(4)])
    again = np.argmin(((x[:, None] - c[None]) ** 2).sum(-1), axis=1)
    np.testing.assert_array_equal(again, assign)


def _cos(u, v):
    return float(np.dot(u, v) / (np.linalg.norm(u) * np.linalg.norm(v)))


def test_pairwise_scores_against_explicit_pair_loop():
    r = np.random.default_rng(3)
    n, d = 7, 5
    fl, fm, fe = (r.standard_normal((n, d)) for _ in range(3))
    anchors = [1, 4]
    members = [0, 2, 3, 5, 6]
    a = {i: max(_cos(fl[i], fl[p]) for p in anchors) for i in range(n)}
    w_mid, w_early = 1.0, 0.5
    expect = []
    for i in members:
        tot = 0.0
        for j in members:
            if j != i:
                tot += (_cos(fl[i], fl[j]) + w_mid * _cos(fm[i], fm[j]) + w_early * _cos(fe[i], fe[j])
                        + a[i] + a[j])
        expect.append(tot / (len(members) - 1))
    ul, um, ue = op.unit_rows(fl), op.unit_rows(fm), op.unit_rows(fe)
    a_arr = op.anchor_similarity(ul, np.array(anchors))
    got = op.pairwise_scores(np.array(members), ul, [um, ue], [w_mid, w_early], a_arr)
    np.testing.assert_allclose(got, expect, rtol=0, atol=1e-12)


def test_pairwise_scores_equal_cluster_sum_identity():
    # sum_{j != i} u_i . u_j = u_i . (sum_j u_j) - 1 for unit rows: the O(n d) form a fast kernel uses.
    r = np.random.default_rng(4)
    n, d = 40, 16
    fl, fm = r.standard_normal((n, d)), r.standard_normal((n, d))
    ul, um = op.unit_rows(fl), op.unit_rows(fm)
    a = r.uniform(0, 1, n)
    members = np.arange(3, 31)
    c = len(members)
    sl, sm, sa = ul[members].sum(0), um[members].sum(0), a[members].sum()
    ident = ((ul[members] @ sl - 1) + (um[members] @ sm - 1)) / (c - 1) + a[members] + (sa - a[members]) / (c - 1)
    got = op.pairwise_scores(members, ul, [um], [1.0], a)
    np.testing.assert_allclose(got, ident, rtol=0, atol=1e-12)


def test_single_cluster_no_anchor_is_plain_redundancy_pruning():
    # K = 1 and r = 0: keep the `keep` tokens of lowest mean (final + middle) cosine to the others.
    r = np.random.default_rng(5)
    n, d, keep = 30, 12, 9
    fl = r.standard_normal((n + 1, d))
    fm = r.standard_normal((n + 1, d))
    attn = r.uniform(size=(2, n + 1))
    res = op.prune_tile([fm, fl], attn, has_cls=True, attn_form=0, final_layer=1, keep=keep,
                        n_clusters=1, anchor_ratio=0.0)
    P, M = fl[1:], fm[1:]
    gl = np.array([[_cos(P[i], P[j]) for j in range(n)] for i in range(n)])
    gm = np.array([[_cos(M[i], M[j]) for j in range(n)] for i in range(n)])
    mean_sim = ((gl + gm).sum(1) - 2.0) / (n - 1)
    expect = np.sort(np.argsort(mean_sim, kind="stable")[:keep])
    np.testing.assert_array_equal(res["keep_idx"], expect)
    assert (res["kind"][expect] == 2).all()


def test_bottom_quota_selection_matches_exhaustive_search():
    r = np.random.default_rng(9)
    n, d, keep = 10, 4, 5
    fl, fm = r.standard_normal((n + 1, d)), r.standard_normal((n + 1, d))
    attn = r.uniform(size=(1, n + 1))
    res = op.prune_tile([fm, fl], attn, has_cls=True, attn_form=0, final_layer=1, keep=keep,
                        n_clusters=1, anchor_ratio=0.0)
    s = res["scores"]
    best = min(itertools.combinations(range(n), keep), key=lambda sub: (sum(s[list(sub)]), sub))
    np.testing.assert_array_equal(res["keep_idx"], best)


@pytest.mark.parametrize("keep", [1, 7, 45, 64, 200, 576])
def test_prune_invariants_on_llava_tile(keep):
    v = synth.vision_tiles(11, 1, 576, 64, 2, 4)
    res = op.prune([v["feats"][0], v["feats"][1]], v["attn"], keep=keep, final_layer=1)[0]
    idx = res["keep_idx"]
    assert len(idx) == keep
    assert np.all(np.diff(idx) > 0) and idx[0] >= 0 and idx[-1] < 576
    assert (res["kind"] == 1).sum() == op.n_anchor_tokens(keep, 0.7)
    assert sum(res["quotas"]) == keep - op.n_anchor_tokens(keep, 0.7)
    assert np.isinf(res["scores"][res["kind"] == 1]).all()
    assert (res["cluster"][res["kind"] == 1] == -1).all()


def test_anchors_are_the_most_attended_tokens():
    v = synth.vision_tiles(12, 1, 576, 32, 2, 8)
    res = op.prune(v["feats"], v["attn"], keep=64, final_layer=1)[0]
    a = v["attn"][0].astype(np.float64)[:, 1:].mean(0)
    anchors = np.flatnonzero(res["kind"] == 1)
    assert a[anchors].min() > np.delete(a, anchors).max()


def test_planted_inputs_are_well_conditioned_for_some_seeds():
    ok = 0
    for seed in range(20260001, 20260013):
        v = synth.vision_tiles(seed, 1, 576, 256, 3, 8)
        res = op.prune(v["feats"], v["attn"], keep=64, final_layer=2)[0]
        ok += op.well_conditioned(res)
    assert ok >= 2


# ---- received attention from full maps (§4.1.1 without [CLS]; the Qwen PatchMerger reading) ----
def _softmax_maps(rng, h, n_q, n_k):
    z = rng.standard_normal((h, n_q, n_k)) * 2.0
    e = np.exp(z - z.max(axis=2, keepdims=True))
    return e / e.sum(axis=2, keepdims=True)


def test_received_attention_conserves_mass_on_non_square_maps():
    # every query row of a softmax map sums to one, so the mean over queries of the attention each
    # key receives sums to one per head (a reduction over the key axis instead would sum to
    # n_q / n_k here)
    rng = np.random.default_rng(1)
    a = _softmax_maps(rng, 3, 7, 12)
    r = op.received_attention(a)
    assert r.shape == (3, 12)
    np.testing.assert_allclose(r.sum(axis=1), 1.0, rtol=0, atol=1e-12)
    g = op.merge_groups_2x2(2, 6)  # the 12 keys as a 2 x 6 grid: three merged tokens
    np.testing.assert_allclose(op.received_attention(a, g).sum(axis=1), 1.0, rtol=0, atol=1e-12)


def test_received_attention_closed_forms():
    n = 24
    uniform = np.full((2, 10, n), 1.0 / n)
    np.testing.assert_allclose(op.received_attention(uniform), 1.0 / n, rtol=1e-15)
    g = op.merge_groups_2x2(4, 6)
    np.testing.assert_allclose(op.received_attention(uniform, g), 4.0 / n, rtol=1e-15)
    one_hot = np.zeros((1, 5, n))
    one_hot[0, :, 13] = 1.0  # every query attends to key 13 only
    r = op.received_attention(one_hot, g)[0]
    owner = [j for j, members in enumerate(g) if 13 in members]
    assert owner == [3]  # key 13 = grid (2, 1): post-merger token (1, 0) of a 2 x 3 post grid
    expect = np.zeros(len(g))
    expect[3] = 1.0
    np.testing.assert_array_equal(r, expect)


def test_received_attention_ignores_query_order():
    rng = np.random.default_rng(2)
    a = _softmax_maps(rng, 2, 9, 9)
    perm = rng.permutation(9)
    np.testing.assert_allclose(op.received_attention(a[:, perm, :]), op.received_attention(a),
                               rtol=1e-13)


def test_merge_groups_2x2_partition_the_grid_into_blocks():
    g = op.merge_groups_2x2(4, 6)
    assert g[0] == [0, 1, 6, 7] and g[1] == [2, 3, 8, 9] and g[3] == [12, 13, 18, 19]
    flat = sorted(i for members in g for i in members)
    assert flat == list(range(24))


# ---- ablation variants of the MSV-Prune table (K, middle-layer and anchor terms, sim kinds) ----
def _sim_brute(x, y, kind):
    """One pair's similarity computed through library routines, not the oracle's formulas."""
    from scipy.spatial.distance import sqeuclidean
    from scipy.special import softmax
    from scipy.stats import entropy
    if kind == "cos":
        return _cos(x, y)
    if kind == "mse":
        return -sqeuclidean(x, y) / len(x)
    return -float(entropy(softmax(x), softmax(y)))


@pytest.mark.parametrize("kind", ["cos", "mse", "kl"])
def test_similarity_kinds_against_library_routines(kind):
    r = np.random.default_rng(21)
    a, b = r.standard_normal((5, 9)), 2.0 * r.standard_normal((4, 9))
    expect = [[_sim_brute(a[i], b[j], kind) for j in range(4)] for i in range(5)]
    np.testing.assert_allclose(op.similarity(a, b, kind), expect, rtol=0, atol=1e-12)


def test_similarity_kinds_invariances():
    r = np.random.default_rng(22)
    a, b = r.standard_normal((6, 8)), r.standard_normal((5, 8))
    base = {k: op.similarity(a, b, k) for k in op.SIM_KINDS}
    # cosine: positive scaling of any row; MSE: one translation of all rows; KL (of softmaxes): a
    # constant added to any row
    s = r.uniform(0.5, 3.0, (6, 1))
    np.testing.assert_allclose(op.similarity(a * s, b, "cos"), base["cos"], atol=1e-12)
    t = r.standard_normal(8)
    np.testing.assert_allclose(op.similarity(a + t, b + t, "mse"), base["mse"], atol=1e-12)
    c = r.standard_normal((6, 1))
    np.testing.assert_allclose(op.similarity(a + c, b, "kl"), base["kl"], atol=1e-12)
    # a row compared with itself: cosine 1, no distance, no divergence; others never exceed that
    for k, top in (("cos", 1.0), ("mse", 0.0), ("kl", 0.0)):
        g = op.similarity(a, a, k)
        np.testing.assert_allclose(np.diag(g), top, atol=1e-12)
        assert (g <= top + 1e-12).all()


@pytest.mark.parametrize("kind,use_final,use_anchor", [
    ("cos", False, True), ("cos", True, False), ("mse", True, True), ("kl", True, True),
    ("mse", False, False), ("kl", True, False)])
def test_ablated_pairwise_scores_against_explicit_pair_loop(kind, use_final, use_anchor):
    r = np.random.default_rng(23)
    n, d = 8, 6
    fl, fm = r.standard_normal((n, d)), r.standard_normal((n, d))
    anchors = [2, 6]
    members = [0, 1, 3, 4, 7]
    a = {i: max(_sim_brute(fl[i], fl[p], kind) for p in anchors) for i in range(n)}
    expect = []
    for i in members:
        tot = 0.0
        for j in members:
            if j != i:
                tot += ((_sim_brute(fl[i], fl[j], kind) if use_final else 0.0)
                        + 0.75 * _sim_brute(fm[i], fm[j], kind)
                        + ((a[i] + a[j]) if use_anchor else 0.0))
        expect.append(tot / (len(members) - 1))
    a_arr = op.anchor_similarity(fl, np.array(anchors), kind)
    got = op.pairwise_scores(np.array(members), fl, [fm], [0.75], a_arr, kind=kind,
                             use_final_sim=use_final, use_anchor_sim=use_anchor)
    np.testing.assert_allclose(got, expect, rtol=0, atol=1e-12)


@pytest.mark.parametrize("kind", ["cos", "mse", "kl"])
def test_outlier_is_kept_over_near_duplicates(kind):
    # ten near-copies of one row and one unrelated row, one cluster, no anchors, keep 1: the
    # unrelated row is the least redundant under every similarity kind
    r = np.random.default_rng(24)
    d = 16
    base = r.standard_normal(d)
    rows = [base + 0.05 * r.standard_normal(d) for _ in range(10)]
    rows.insert(7, -base + 0.5 * r.standard_normal(d))
    f = np.vstack([np.zeros(d), np.array(rows)])  # row 0 is [CLS]
    attn = r.uniform(size=(1, 12))
    res = op.prune_tile([f, f], attn, has_cls=True, attn_form=0, final_layer=1, keep=1, n_clusters=1,
                        anchor_ratio=0.0, sim=kind)
    np.testing.assert_array_equal(res["keep_idx"], [7])


def test_without_anchor_term_anchor_features_do_not_matter():
    v = synth.vision_tiles(25, 1, 144, 32, 2, 4)
    feats = [f[0].copy() for f in v["feats"]]
    kw = dict(has_cls=True, attn_form=0, final_layer=1, keep=40, anchor_ratio=0.5)
    ref = op.prune_tile(feats, v["attn"][0], use_anchor_sim=False, **kw)
    anchors = np.flatnonzero(ref["kind"] == 1)
    moved = [f.copy() for f in feats]
    for f in moved:
        f[1 + anchors] = np.random.default_rng(26).standard_normal((len(anchors), f.shape[1]))
    got = op.prune_tile(moved, v["attn"][0], use_anchor_sim=False, **kw)
    np.testing.assert_array_equal(got["keep_idx"], ref["keep_idx"])
    np.testing.assert_array_equal(got["scores"], ref["scores"])
    # with the anchor term the same move changes the scores
    with_term = op.prune_tile(feats, v["attn"][0], **kw)
    moved_term = op.prune_tile(moved, v["attn"][0], **kw)
    assert not np.allclose(with_term["scores"][ref["kind"] != 1], moved_term["scores"][ref["kind"] != 1])


def test_only_middle_layer_scores_ignore_final_layer_beyond_clustering():
    # without the final-layer term, F^L enters only through K = 1 clustering (trivial) and the
    # anchor bracket (dropped too): the scores are those of the middle layer alone
    r = np.random.default_rng(27)
    n, d = 20, 8
    fm, fl = r.standard_normal((n + 1, d)), r.standard_normal((n + 1, d))
    attn = r.uniform(size=(1, n + 1))
    kw = dict(has_cls=True, attn_form=0, final_layer=1, keep=6, n_clusters=1, anchor_ratio=0.0,
              use_final_sim=False)
    a = op.prune_tile([fm, fl], attn, **kw)
    b = op.prune_tile([fm, r.standard_normal((n + 1, d))], attn, **kw)
    np.testing.assert_array_equal(a["scores"], b["scores"])
    g = np.array([[_cos(fm[1 + i], fm[1 + j]) for j in range(n)] for i in range(n)])
    np.testing.assert_allclose(a["scores"], (g.sum(1) - 1.0) / (n - 1), atol=1e-12)


@pytest.mark.parametrize("K", [1, 2, 8])
def test_cluster_count_variants_keep_the_budget(K):
    v = synth.vision_tiles(28, 1, 576, 32, 2, 4)
    res = op.prune(v["feats"], v["attn"], keep=64, final_layer=1, n_clusters=K)[0]
    assert len(res["keep_idx"]) == 64
    assert sum(res["quotas"]) == 64 - op.n_anchor_tokens(64, 0.7)
    c = res["cluster"][res["kind"] != 1]
    assert c.min() >= 0 and c.max() < K
    assert all(q >= 1 for q, sz in zip(res["quotas"], res["sizes"]) if sz > 0)
