"""CPU oracle of MSV-Prune, multi-layer semantic visual-token pruning (§4.1, Eq. 1-3, Alg. 1 stage 1).

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may import
this module. It shares no code with the CUDA path. It is plain and slow, and computes in fp64.

The paper is silent or ambiguous on several points. The readings taken here (ties, roundings,
K-means initialisation, the per-token reading of the pairwise score) are the ones the CUDA path
implements, and each is stated where it is used.

Pinned by tests/test_oracle_prune.py against brute force, closed forms and invariants.
"""
from __future__ import annotations

from fractions import Fraction

import numpy as np


def attention_importance(attn_tile: np.ndarray, form: int) -> np.ndarray:
    """a_v for one tile: the head-mean of the encoder self-attention (§4.1.1).

    form 0 (CLIP-like): attn_tile is the [CLS] row per head, [H][1+n]. Column 0 (CLS attending to
    itself) is not a patch and is dropped. form 1 (no CLS): attn_tile is the attention each patch
    receives per head, [H][n].
    """
    a = np.asarray(attn_tile, dtype=np.float64)
    if form == 0:
        a = a[:, 1:]
    return a.mean(axis=0)


def received_attention(maps: np.ndarray, groups=None) -> np.ndarray:
    """Received-attention form [H][n_out] from full self-attention maps [H][n_q][n_k] (§4.1.1:
    without a [CLS] token, the importance of a patch is the mean attention it receives).

    R[h, i] = (1 / n_q) * sum over query rows q of maps[h, q, i].

    groups (optional): for encoders with a patch merger (§Implementation details: Qwen's
    PatchMerger), a list over post-merger tokens of the pre-merger token indices each one merges.
    The post-merger token receives the attention its members receive, summed: merging keys merges
    their probability mass (reading: the paper states that importance is computed on post-merger
    tokens but not how attention is carried through the merger). Without groups, n_out = n_k.
    """
    a = np.asarray(maps, dtype=np.float64)
    h, n_q, n_k = a.shape
    r = np.zeros((h, n_k))
    for q in range(n_q):  # explicit sum over the query rows
        r += a[:, q, :]
    r /= n_q
    if groups is None:
        return r
    out = np.zeros((h, len(groups)))
    for j, members in enumerate(groups):
        for i in members:
            out[:, j] += r[:, i]
    return out


def merge_groups_2x2(rows: int, cols: int):
    """Pre-merger token indices of each post-merger token for a 2 x 2 spatial merger over a
    rows x cols patch grid (row-major, both even): post token (y, x) merges patches (2y + dy,
    2x + dx), dy, dx in {0, 1}, listed in ascending index order."""
    groups = []
    for y in range(rows // 2):
        for x in range(cols // 2):
            groups.append(sorted((2 * y + dy) * cols + 2 * x + dx for dy in (0, 1) for dx in (0, 1)))
    return groups


def n_anchor_tokens(keep: int, anchor_ratio: float) -> int:
    """N_anc = round(keep * r), half away from zero, evaluated in double (§4.1, Eq. 1 budget n R r).

    keep = n R is the retained count. N_cmp = keep - N_anc, so the two parts always add up to keep.
    """
    return int(np.floor(keep * anchor_ratio + 0.5))


def select_anchors(a_v: np.ndarray, n_anc: int) -> np.ndarray:
    """Eq. 1: the anchor set is the n_anc tokens of largest a_v.

    The threshold form (the smallest tau with at most n R r scores >= tau) names exactly this
    top-n_anc set. Equal scores are broken toward the lower token index. Returns indices ascending.
    """
    n = len(a_v)
    order = sorted(range(n), key=lambda i: (-a_v[i], i))
    return np.array(sorted(order[:n_anc]), dtype=np.int64)


def unit_rows(f: np.ndarray) -> np.ndarray:
    """Rows divided by their Euclidean norm, so that dot products are cosine similarities."""
    f = np.asarray(f, dtype=np.float64)
    return f / np.sqrt((f * f).sum(axis=1, keepdims=True))


SIM_KINDS = ("cos", "mse", "kl")


def log_softmax_rows(f: np.ndarray) -> np.ndarray:
    """log of the softmax of every row over the feature dimension (shifted by the row maximum)."""
    f = np.asarray(f, dtype=np.float64)
    z = f - f.max(axis=1, keepdims=True)
    return z - np.log(np.exp(z).sum(axis=1, keepdims=True))


def similarity(a: np.ndarray, b: np.ndarray, kind: str = "cos") -> np.ndarray:
    """sim(F_i, F_j) of Eq. 3 for every row i of a and row j of b, as an [len(a)][len(b)] matrix.

    cos: the cosine similarity, the paper's choice.
    mse, kl: the ablation of the MSV-Prune table, part (c), that puts the mean squared error or the
    Kullback-Leibler divergence in place of the cosine. Both measure dissimilarity, so they enter
    Eq. 3 negated: a larger value still means more alike, and the N_k lowest-scoring tokens of a
    cluster are still its least redundant ones (reading: the paper names only the replacement).
      mse: -(1/d) sum_k (a_ik - b_jk)^2
      kl:  -KL(P_i || Q_j) = -sum_k P_ik (log P_ik - log Q_jk), with P_i and Q_j the softmax of the
           rows over the feature dimension (reading: features are not distributions, and the
           softmax is what makes them ones).
    """
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    if kind == "cos":
        return unit_rows(a) @ unit_rows(b).T
    out = np.empty((len(a), len(b)))
    if kind == "mse":
        for i in range(len(a)):  # one row of the matrix at a time (bounded memory)
            out[i] = -((b - a[i]) ** 2).mean(axis=1)
        return out
    if kind == "kl":
        la, lb = log_softmax_rows(a), log_softmax_rows(b)
        for i in range(len(a)):
            out[i] = -(np.exp(la[i]) * (la[i] - lb)).sum(axis=1)
        return out
    raise ValueError(f"unknown similarity kind {kind!r}")


def anchor_similarity(f_final: np.ndarray, anchors: np.ndarray, kind: str = "cos") -> np.ndarray:
    """max over anchors p of sim(F^L_i, F^L_p), for every token i (Eq. 3, second bracket).

    With no anchors (r = 0) the term is absent and 0 is returned.
    """
    if len(anchors) == 0:
        return np.zeros(len(f_final))
    f_final = np.asarray(f_final, dtype=np.float64)
    return similarity(f_final, f_final[anchors], kind).max(axis=1)


def kmeans(x: np.ndarray, k: int, iters: int):
    """K-means (Lloyd) on the rows of x, the final-layer features of the non-anchor tokens (§4.1.2).

    The paper names K-means on F^L and nothing more. Readings taken here:
    * initial centroids are the rows at positions floor(j * m / K), j = 0..K-1, of the non-anchor
      tokens in ascending token order;
    * the distance is the squared Euclidean distance sum_d (x_d - c_d)^2;
    * each step assigns every point to its nearest centroid (ties to the lower cluster id);
    * at most `iters` assignment steps, stopping early once the assignment repeats;
    * each assignment step is followed by a centroid update (mean of the members); an empty
      cluster keeps its previous centroid.

    Returns (assignment [m], min relative margin (second - best) / best over all steps and points).
    """
    x = np.asarray(x, dtype=np.float64)
    m = len(x)
    if m == 0:
        return np.zeros(0, dtype=np.int64), np.inf
    c = np.stack([x[(j * m) // k] for j in range(k)])
    assign = None
    margin = np.inf
    for _ in range(iters):
        d2 = ((x[:, None, :] - c[None, :, :]) ** 2).sum(axis=2)
        new = np.argmin(d2, axis=1)
        if k > 1:
            srt = np.sort(d2, axis=1)
            margin = min(margin, float(((srt[:, 1] - srt[:, 0]) / np.maximum(srt[:, 0], 1e-300)).min()))
        if assign is not None and np.array_equal(new, assign):
            break
        assign = new
        for j in range(k):
            members = x[assign == j]
            if len(members):
                c[j] = members.mean(axis=0)
    return assign, margin


def _round_half_away(fr: Fraction) -> int:
    return int((fr * 2 + 1) // 2)  # fr >= 0 here


def cluster_quotas(sizes, n_cmp: int):
    """Eq. 2: N_k = max(1, round(N_cmp |C_k| / sum_j |C_j|)), made to add up to N_cmp.

    Eq. 2 alone need not sum to N_cmp, and its floor of 1 cannot hold when N_cmp is smaller than the
    number of non-empty clusters. Reading taken (exact rational arithmetic):
    * q_k = N_cmp |C_k| / sum|C|; N_k = max(1, round_half_away(q_k)) for non-empty clusters, 0 for
      empty ones, capped at |C_k|;
    * if N_cmp < number of non-empty clusters: one each to the largest clusters (ties to lower k);
    * if the sum is short: passes over the clusters in descending fractional part of q_k (ties to
      lower k) add 1 to each cluster that has room, until the sum is N_cmp;
    * if the sum is over: passes in ascending fractional part (ties to higher k) take 1 from each
      cluster with N_k > 1, until the sum is N_cmp.
    """
    sizes = [int(s) for s in sizes]
    K = len(sizes)
    total = sum(sizes)
    quota = [0] * K
    if n_cmp <= 0 or total == 0:
        return quota
    nonempty = [k for k in range(K) if sizes[k] > 0]
    if n_cmp < len(nonempty):
        for k in sorted(nonempty, key=lambda k: (-sizes[k], k))[:n_cmp]:
            quota[k] = 1
        return quota
    q = [Fraction(n_cmp * sizes[k], total) for k in range(K)]
    frac = [qk - (qk.numerator // qk.denominator) for qk in q]
    for k in nonempty:
        quota[k] = min(sizes[k], max(1, _round_half_away(q[k])))
    while sum(quota) < n_cmp:
        for k in sorted(range(K), key=lambda k: (-frac[k], k)):
            if sum(quota) < n_cmp and quota[k] < sizes[k]:
                quota[k] += 1
    while sum(quota) > n_cmp:
        for k in sorted(range(K), key=lambda k: (frac[k], -k)):
            if sum(quota) > n_cmp and quota[k] > 1:
                quota[k] -= 1
    return quota


def pairwise_scores(members, feats_final, feats_other, other_weights, a_anchor, *, kind="cos",
                    use_final_sim=True, use_anchor_sim=True):
    """Eq. 3 for the tokens of one cluster, reduced to one score per token.

    S_ij = sim(F^L_i, F^L_j) + sim(F^M_i, F^M_j) + max_p sim(F^L_i, F^L_p) + max_p sim(F^L_j, F^L_p).
    The paper selects the N_k lowest-scoring tokens of each cluster from this pairwise score; the
    per-token score read here is the mean of S_ij over the other members j != i of the cluster. The
    intra-cluster term sums every tapped non-final layer with its weight (one middle layer with
    weight 1 in the paper). A singleton cluster has no pair; its token scores 2 * a_i.

    Ablations of the MSV-Prune table: `kind` replaces the cosine (see similarity); without the
    final-layer term (use_final_sim False: "only middle layer tokens" in the intra-cluster part)
    and without the anchor bracket (use_anchor_sim False). A zero weight of the middle layer gives
    "without middle layer tokens".

    Computed literally: the full |C| x |C| matrix of S_ij, diagonal excluded.
    """
    members = np.asarray(members)
    c = len(members)
    a = a_anchor[members] if use_anchor_sim else np.zeros(c)
    if c == 1:
        return 2.0 * a
    s = np.zeros((c, c))
    if use_final_sim:
        f = feats_final[members]
        s = s + similarity(f, f, kind)
    for w, fo in zip(other_weights, feats_other):
        v = fo[members]
        s = s + w * similarity(v, v, kind)
    s = s + a[:, None] + a[None, :]
    np.fill_diagonal(s, 0.0)
    return s.sum(axis=1) / (c - 1)


def prune_tile(feats, attn_tile, *, has_cls: bool, attn_form: int, final_layer: int, keep: int,
               n_clusters: int = 4, kmeans_iters: int = 10, anchor_ratio: float = 0.7,
               layer_weight=None, sim: str = "cos", use_final_sim: bool = True,
               use_anchor_sim: bool = True):
    """MSV-Prune of one tile (Alg. 1 stage 1): anchors, clustering, scoring, per-cluster selection.

    sim, use_final_sim, use_anchor_sim: the ablations of pairwise_scores (the paper's method is
    cos, True, True); n_clusters = 1 is the ablation without semantic clustering.

    feats: list over tapped layers of [n_tok][d] arrays (row 0 is [CLS] when has_cls, never kept).
    Returns a dict with keep_idx (ascending patch indices, length keep), kind (0 dropped, 1 anchor,
    2 complementary), cluster (-1 for anchors), scores (Eq. 3 per-token score; +inf for anchors),
    quotas, a_v, anchor_sim, and margins of every discrete decision (anchor cut, K-means, per-cluster
    cuts) for input conditioning.
    """
    off = 1 if has_cls else 0
    patch = [np.asarray(f, dtype=np.float64)[off:] for f in feats]
    n = patch[0].shape[0]
    if not 1 <= keep <= n:
        raise ValueError("keep must lie in [1, n_patch]")
    n_layers = len(patch)
    if layer_weight is None:
        layer_weight = [1.0] * n_layers
    others = [l for l in range(n_layers) if l != final_layer]

    a_v = attention_importance(attn_tile, attn_form)
    n_anc = n_anchor_tokens(keep, anchor_ratio)
    n_cmp = keep - n_anc
    anchors = select_anchors(a_v, n_anc)
    is_anchor = np.zeros(n, dtype=bool)
    is_anchor[anchors] = True
    rest = np.flatnonzero(~is_anchor)

    if sim not in SIM_KINDS:
        raise ValueError(f"unknown similarity kind {sim!r}")
    feats_final = patch[final_layer]
    feats_other = [patch[l] for l in others]
    a_sim = anchor_similarity(feats_final, anchors, sim) if use_anchor_sim else np.zeros(n)

    assign, km_margin = kmeans(patch[final_layer][rest], n_clusters, kmeans_iters)
    sizes = [int((assign == k).sum()) for k in range(n_clusters)]
    quotas = cluster_quotas(sizes, n_cmp)

    scores = np.full(n, np.inf)
    cluster = np.full(n, -1, dtype=np.int64)
    cluster[rest] = assign
    selected = []
    cut_gap = np.inf
    for k in range(n_clusters):
        members = rest[assign == k]
        if len(members) == 0:
            continue
        s = pairwise_scores(members, feats_final, feats_other, [layer_weight[l] for l in others],
                            a_sim, kind=sim, use_final_sim=use_final_sim,
                            use_anchor_sim=use_anchor_sim)
        scores[members] = s
        order = sorted(range(len(members)), key=lambda j: (s[j], members[j]))
        selected.extend(members[order[:quotas[k]]].tolist())
        if 0 < quotas[k] < len(members):
            cut_gap = min(cut_gap, float(s[order[quotas[k]]] - s[order[quotas[k] - 1]]))

    kind = np.zeros(n, dtype=np.uint8)
    kind[anchors] = 1
    kind[np.array(selected, dtype=np.int64)] = 2
    keep_idx = np.flatnonzero(kind > 0)
    srt = np.sort(a_v)[::-1]
    anchor_gap = float((srt[n_anc - 1] - srt[n_anc]) / srt[n_anc - 1]) if 0 < n_anc < n else np.inf
    return dict(keep_idx=keep_idx, kind=kind, cluster=cluster, scores=scores, quotas=quotas,
                sizes=sizes, a_v=a_v, anchor_sim=a_sim, n_anchor=n_anc,
                margins=dict(anchor_gap=anchor_gap, kmeans=km_margin, cut_gap=cut_gap))


def prune(feats, attn, *, has_cls=True, attn_form=0, final_layer=-1, keep=64, n_clusters=4,
          kmeans_iters=10, anchor_ratio=0.7, layer_weight=None, sim="cos", use_final_sim=True,
          use_anchor_sim=True):
    """MSV-Prune of every tile independently (AnyRes: same rule and budget per tile, §5.1).

    feats: list over tapped layers of [n_tiles][n_tok][d]; attn: [n_tiles][H][n_att].
    """
    final_layer = final_layer % len(feats)
    out = []
    for t in range(attn.shape[0]):
        out.append(prune_tile([f[t] for f in feats], attn[t], has_cls=has_cls, attn_form=attn_form,
                              final_layer=final_layer, keep=keep, n_clusters=n_clusters,
                              kmeans_iters=kmeans_iters, anchor_ratio=anchor_ratio,
                              layer_weight=layer_weight, sim=sim, use_final_sim=use_final_sim,
                              use_anchor_sim=use_anchor_sim))
    return out


def well_conditioned(result, gap: float = 1e-3) -> bool:
    """True when every discrete decision of a prune_tile result has a margin above `gap`.

    Used to pick seeded inputs on which an fp32 implementation and this fp64 oracle must agree
    index for index: anchor cut (relative a_v gap), K-means (relative distance margin), and the
    per-cluster selection cuts (absolute score gap).
    """
    m = result["margins"]
    return m["anchor_gap"] > gap and m["kmeans"] > gap and m["cut_gap"] > gap
