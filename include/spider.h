/*
 * spider.h - C ABI of libspider.so, SPIDER's accelerated multimodal prefill on one GB300 (sm_103a).
 *
 * Two stages, as in Alg. 1 of the paper:
 *   1. MSV-Prune (Sec. 4.1, Eq. 1-3): score, select and compact the visual tokens of each tile.
 *   2. Decoder prefill with adaptive sub-layer skipping (Sec. 3.2, 4.2-4.3): every layer's attention
 *      and FFN sub-layers run or are bypassed per token, following a skip mask.
 *
 * Conventions for every entry point:
 *   - Pointers marked (dev) are device memory of the current CUDA device; (host) are host memory.
 *     bf16 data is passed as uint16_t bit patterns. Matrices are row-major.
 *   - The caller owns every buffer. Work is enqueued on `stream` (a cudaStream_t, NULL = legacy
 *     default stream) and is asynchronous unless stated otherwise.
 *   - spd_prune, spd_project, spd_prefill and spd_linear allocate nothing: they run in a
 *     caller-provided workspace whose size the matching *_workspace_size call returns. A workspace
 *     must not be shared by calls that may overlap on the GPU.
 *   - Every call returns SPD_OK (0) or a negative spd_status. Argument errors are detected on the
 *     host before any launch and leave the device untouched; spd_last_error() describes the last
 *     failure of the calling thread. Device-side failures (a bounded wait that gave up) are
 *     recorded in the workspace's status word, read back by spd_workspace_status().
 */
#ifndef SPIDER_H
#define SPIDER_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  SPD_OK = 0,
  SPD_EINVAL = -1,       /* invalid argument or configuration (checked on the host) */
  SPD_ENOSPC = -2,       /* workspace smaller than the size query returned */
  SPD_ECUDA = -3,        /* a CUDA runtime/driver call failed */
  SPD_ETIMEOUT = -4,     /* a bounded device-side wait gave up (kernel returned early) */
  SPD_EUNSUPPORTED = -5  /* shape outside what the kernels implement (e.g. head_dim) */
} spd_status;

#define SPD_MAX_FEAT_LAYERS 4
#define SPD_MAX_CLUSTERS 16

/* Message of the last failed call on this thread (static storage, never NULL). */
const char* spd_last_error(void);

/* Reads and clears the device status word at the start of a workspace (synchronises `stream`).
 * *status receives SPD_OK or the first device-side failure recorded since the last read. */
int spd_workspace_status(void* ws, void* stream, int* status);

/* Failure-detection self-test (no counterpart in the paper): launches one CTA whose thread waits,
 * with the same bounded wait every pipelined kernel here uses, on a barrier that nothing ever
 * arrives on. After `budget_cycles` SM clock cycles the wait gives up and records SPD_ETIMEOUT in
 * the status word of `ws` (at least 4 bytes of device memory). No fault, trap or hang: the
 * context stays usable. Asynchronous; read the result with spd_workspace_status. */
int spd_selftest_bounded_wait(void* ws, long long budget_cycles, void* stream);

/* Deterministic mode (library-wide; no counterpart in the paper). With on != 0, every GEMM sums
 * each output element in a fixed order: K-split tiles store per-CTA fp32 partials that the tile's
 * last CTA adds in CTA order, and residual updates of the fp32 stream are one read-modify-write per
 * element. Repeated calls on the same inputs then give bit-identical results. With on = 0 (the
 * default), split partial sums and residual updates are fire-and-forget fp32 reductions at L2,
 * whose order varies, so the last bits (and, through bf16 roundings downstream, a bf16 unit) may
 * differ between runs. Takes effect for launches enqueued after the call; returns SPD_OK. */
int spd_set_deterministic(int on);

/* Kernel-class tracing (no counterpart in the paper; measurement support). spd_trace_enable(n)
 * starts recording up to n launches: every launch of the library is bracketed by a CUDA event pair
 * on its stream and tagged with its class and algorithmic work; n <= 0 stops recording.
 * spd_trace_read synchronises on the recorded events and returns, for one class
 * (SPD_TRACE_GEMM, _ATTN, _ROWS, _PRUNE), the launch count, summed device milliseconds, and summed
 * algorithmic flops and HBM bytes (the operation's own: operands read once, results written once). */
#define SPD_TRACE_GEMM 0
#define SPD_TRACE_ATTN 1
#define SPD_TRACE_ROWS 2
#define SPD_TRACE_PRUNE 3
int spd_trace_enable(int capacity);
int spd_trace_read(int cls, long long* launches, double* ms, double* flops, double* bytes);

/* Launch stamps (measurement support, no counterpart in the paper): spd_stamp_enable(n) starts
 * stamping up to n launches of the GEMM, attention and RMSNorm kernels without adding any stream
 * operation between launches: each stamped kernel records, in device memory, the globaltimer time
 * of its first CTA past the grid dependency wait and of its last CTA's end. n <= 0 stops. The
 * intervals of successive kernels of a stream do not overlap (a kernel passes its wait only after
 * its predecessor completed), so a class's summed time never exceeds the wall time of the work.
 * spd_stamp_read synchronises the device and returns for one class (SPD_TRACE_*) the launch count,
 * summed milliseconds and summed algorithmic flops and bytes, as spd_trace_read. Not thread-safe
 * with respect to concurrent library calls from other threads (the slots are taken in call
 * order). Errors: SPD_ECUDA. */
int spd_stamp_enable(int capacity);
int spd_stamp_read(int cls, long long* launches, double* ms, double* flops, double* bytes);
/* Stamp k (0-based, in launch order since spd_stamp_enable): class, start and end (globaltimer ns;
 * end < start when the launch did not run), algorithmic flops and bytes. Synchronises the device.
 * Errors: SPD_EINVAL when fewer than k + 1 launches were stamped; SPD_ECUDA. */
int spd_stamp_launch(int k, int* cls, unsigned long long* start_ns, unsigned long long* end_ns,
                     double* flops, double* bytes);

/* ------------------------------------------------------------------------------------------ */
/* Stage 1: MSV-Prune (Sec. 4.1)                                                                */
/* ------------------------------------------------------------------------------------------ */

typedef struct {
  int n_tiles;      /* independent tiles (images, or AnyRes crops pruned separately, Sec. 5.1) */
  int n_tok;        /* rows per tile in the feature arrays, including the [CLS] row if has_cls */
  int has_cls;      /* 1: row 0 of every tile is [CLS]; it is never kept */
  int d_feat;       /* feature width, a multiple of 4, at most 4096 */
  int n_layers;     /* tapped encoder layers, 1..SPD_MAX_FEAT_LAYERS */
  int final_layer;  /* index of the tapped layer that is F^L (final-layer features) */
  int n_heads;      /* encoder attention heads in `attn` */
  int attn_form;    /* 0: [CLS] attention row per head, [n_heads][n_tok] (column 0 = CLS->CLS);
                       1: attention received by each patch per head, [n_heads][n_tok - has_cls] */
  int keep;         /* tokens kept per tile, 1..n_patch (n_patch = n_tok - has_cls, <= 4096) */
  int n_clusters;   /* K of the coarse clustering, 1..SPD_MAX_CLUSTERS (paper default 4) */
  int kmeans_iters; /* maximum Lloyd assignment steps, >= 1 (stops early on a repeated assignment) */
  double anchor_ratio; /* r in [0, 1]; N_anc = floor(keep * r + 0.5), N_cmp = keep - N_anc */
  float layer_weight[SPD_MAX_FEAT_LAYERS]; /* weight of each non-final layer's intra-cluster cosine
                       term in the score; 1 everywhere reproduces Eq. 3 (entry of final_layer unused);
                       0 for the middle layer is the ablation without middle-layer tokens */
  int sim_kind;     /* sim() of Eq. 3: SPD_SIM_COS (the paper's) or an ablation below */
  int ablate;       /* bit set of SPD_PRUNE_NO_* below; 0 = Eq. 3 as printed */
} spd_prune_cfg;

/* Similarity kinds of Eq. 3 (the MSV-Prune ablation table, part (c)). The two dissimilarities enter
 * negated, so that the N_k lowest-scoring tokens stay the least redundant ones:
 *   SPD_SIM_COS  cos(F_i, F_j)
 *   SPD_SIM_MSE  -(1/d) sum_c (F_i,c - F_j,c)^2
 *   SPD_SIM_KL   -KL(softmax(F_i) || softmax(F_j)), softmax over the feature dimension.
 * Ablation bits: SPD_PRUNE_NO_FINAL_SIM drops sim(F^L_i, F^L_j) from the intra-cluster bracket
 * (with a middle layer: "only middle layer tokens"; with a zero middle weight as well: no
 * intra-cluster term); SPD_PRUNE_NO_ANCHOR_SIM drops the bracket of similarities to the anchors.
 * n_clusters = 1 is the ablation without semantic clustering. */
#define SPD_SIM_COS 0
#define SPD_SIM_MSE 1
#define SPD_SIM_KL 2
#define SPD_PRUNE_NO_FINAL_SIM 1
#define SPD_PRUNE_NO_ANCHOR_SIM 2

/* Bytes of device workspace spd_prune needs for `cfg` (0 if cfg is invalid). */
size_t spd_prune_workspace_size(const spd_prune_cfg* cfg);

/* Number of kernels spd_prune enqueues for `cfg` on the current device (measurement support, no
 * counterpart in the paper): 4 where the K-means kernel also scores, selects and compacts (rows
 * resident in shared memory, cosine similarity), else 6; one less without the anchor maximum
 * (no anchors, or the ablation without it), one less without non-anchor tokens. Negative
 * spd_status on an invalid configuration. */
int spd_prune_launches(const spd_prune_cfg* cfg);

/* MSV-Prune of every tile (Sec. 4.1; Alg. 1 stage 1):
 *   a_v = head-mean of the attention (Sec. 4.1.1); anchors = the N_anc tokens of largest a_v
 *   (Eq. 1, ties to the lower index); K-means (Lloyd, squared Euclidean, seeds at the quantiles
 *   floor(k m / K) of the m non-anchor tokens in index order, empty clusters keep their centroid)
 *   on F^L of the non-anchor tokens; quotas N_k by Eq. 2 made to sum to N_cmp; per-token score =
 *   mean over the other members j of the cluster of S_ij (Eq. 3); in each cluster the N_k
 *   lowest-scoring tokens (ties to the lower index) join the anchors; kept indices ascending.
 *   sim_kind and ablate select the ablation variants of Eq. 3 described above.
 * feats    (host array of n_layers dev pointers) each [n_tiles][n_tok][d_feat] fp32.
 * attn     (dev) fp32, [n_tiles][n_heads][n_tok] (form 0) or [n_tiles][n_heads][n_patch] (form 1).
 * keep_idx (dev) int32 [n_tiles][keep]: kept patch indices (0-based, CLS excluded), ascending.
 * kind     (dev, may be NULL) uint8 [n_tiles][n_patch]: 0 dropped, 1 anchor, 2 complementary.
 * cluster  (dev, may be NULL) int8 [n_tiles][n_patch]: K-means cluster, -1 for anchors.
 * scores   (dev, may be NULL) fp32 [n_tiles][n_patch]: per-token Eq. 3 score, +inf for anchors.
 * All pointers 16-byte aligned. Errors: SPD_EINVAL, SPD_ENOSPC, SPD_ECUDA. */
int spd_prune(const spd_prune_cfg* cfg, const float* const* feats, const float* attn,
              int32_t* keep_idx, uint8_t* kind, int8_t* cluster, float* scores,
              void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes of spd_received_attention. */
size_t spd_received_attention_workspace_size(int n_maps, int n_q, int n_k);

/* The received-attention input form of spd_prune (attn_form 1) from full self-attention maps
 * (Sec. 4.1.1: for an encoder without a [CLS] token a patch's importance is the mean attention it
 * receives), per map m (tile x head):
 *   R[m][i] = (1 / n_q) sum over query rows q of maps[m][q][i],
 * optionally carried through a patch merger whose post-merger token j merges pre-merger tokens
 * group_members[group_start[j] .. group_start[j+1]) (ascending): out[m][j] = sum of R[m][i] over
 * the members (merging keys merges their attention mass; the paper computes importance on the
 * post-merger tokens but does not state the aggregation - this is the library's reading).
 * maps (dev) fp32 [n_maps][n_q][n_k], 16-byte aligned, n_k a multiple of 4; group_start (dev)
 * int32 [n_out + 1] and group_members (dev) int32, both NULL for no merger (then n_out = n_k);
 * out (dev) fp32 [n_maps][n_out]. Sums run in a fixed order (bit-identical run to run).
 * Errors: SPD_EINVAL (arguments; a member index outside [0, n_k) is reported through the
 * workspace's status word), SPD_ENOSPC. */
int spd_received_attention(const float* maps, int n_maps, int n_q, int n_k, const int32_t* group_start,
                           const int32_t* group_members, int n_out, float* out, void* ws,
                           size_t ws_bytes, void* stream);

/* Gathers the kept rows of a per-tile payload (e.g. F^L) into packed bf16 rows for the projector:
 * dst[t * keep + j][:] = bf16(src[t][row_offset + idx[t][j]][:]), round to nearest even.
 * src (dev) fp32 [n_tiles][n_tok][d]; idx (dev) int32 [n_tiles][keep]; dst (dev) bf16
 * [n_tiles * keep][d]. d a multiple of 4. Indices outside [0, n_tok - row_offset) are skipped and
 * reported as SPD_EINVAL through the status word of `ws` (may be NULL: no report). */
int spd_gather_rows_bf16(const float* src, int n_tiles, int n_tok, int d, int row_offset,
                         const int32_t* idx, int keep, uint16_t* dst, void* ws, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Stage 2: decoder prefill with sub-layer skipping (Sec. 3.2, 4.2, 4.3)                        */
/* ------------------------------------------------------------------------------------------ */

typedef struct {
  int n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ffn, vocab;
  float rope_theta;  /* rotary base; pairs (j, j + head_dim/2) rotate by pos * theta^(-2j/head_dim) */
  float rms_eps;     /* RMSNorm epsilon */
  int d_vis;         /* projector input width (vision features); 0 = no projector */
  int d_proj;        /* projector hidden width */
} spd_model_cfg;

/* One decoder layer's weights, bf16 (dev), [out][in] row-major (y = x W^T). */
typedef struct {
  const uint16_t* attn_norm; /* [d_model] RMSNorm gain before attention */
  const uint16_t* wq;        /* [n_heads * head_dim][d_model] */
  const uint16_t* wk;        /* [n_kv_heads * head_dim][d_model] */
  const uint16_t* wv;        /* [n_kv_heads * head_dim][d_model] */
  const uint16_t* wo;        /* [d_model][n_heads * head_dim] */
  const uint16_t* ffn_norm;  /* [d_model] */
  const uint16_t* w_gate;    /* [d_ffn][d_model] */
  const uint16_t* w_up;      /* [d_ffn][d_model] */
  const uint16_t* w_down;    /* [d_model][d_ffn] */
} spd_layer_weights;

typedef struct {
  const spd_layer_weights* layers; /* (host) array of n_layers */
  const uint16_t* final_norm;      /* [d_model] */
  const uint16_t* lm_head;         /* [vocab][d_model] */
  const uint16_t* proj_w1;         /* [d_proj][d_vis]   (only if d_vis > 0) */
  const uint16_t* proj_b1;         /* [d_proj] */
  const uint16_t* proj_w2;         /* [d_model][d_proj] */
  const uint16_t* proj_b2;         /* [d_model] */
} spd_model_weights;

typedef struct spd_model spd_model;

/* Copies the weights into a handle, re-laid out for the GEMM kernels (device memory is allocated
 * here, and only here). Synchronous. The caller's weight buffers may be freed afterwards.
 * Requirements: head_dim in {64, 128}; n_heads a multiple of n_kv_heads; d_model, d_ffn, d_vis and
 * d_proj multiples of 8. Errors: SPD_EINVAL, SPD_EUNSUPPORTED, SPD_ECUDA. */
int spd_model_create(const spd_model_cfg* cfg, const spd_model_weights* w, spd_model** out);
void spd_model_destroy(spd_model* m);

/* Expands Alg. 1's per-token plan into per-layer skip bits (host only):
 * a token with admit[i] >= 0 bypasses sub-layer target[i] (1 attention, 2 FFN, 3 both) in every layer
 * l >= admit[i] (the target is frozen at admission, Sec. 4.2). admit -1 = never.
 * mask (host) uint8 [n_layers][n_tokens]: bit 0 skip attention, bit 1 skip FFN. */
int spd_plan_adaptive(int n_layers, int n_tokens, const int16_t* admit, const uint8_t* target,
                      uint8_t* mask);

/* Static sparse-layer replacement (Sec. 3.2): layer l bypasses the sub-layers in layer_mask[l]
 * (same bits) for every token with token_sel[i] != 0 (the visual tokens). Host only. */
int spd_plan_static(int n_layers, int n_tokens, const uint8_t* layer_mask, const uint8_t* token_sel,
                    uint8_t* mask);

/* Workspace bytes of spd_project for up to `rows` visual rows. */
size_t spd_project_workspace_size(const spd_model* m, int rows);

/* LLaVA MLP projector on gathered visual rows: x[out_rows[r]] = bf16(W2 bf16(GELU(W1 v_r + b1)) + b2)
 * (exact erf GELU). vis (dev) bf16 [rows][d_vis]; out_rows (dev) int32 [rows]; x (dev) bf16
 * [*][d_model], the decoder's input sequence. Errors: SPD_EINVAL (no projector), SPD_ENOSPC. */
int spd_project(const spd_model* m, const uint16_t* vis, int rows, const int32_t* out_rows,
                uint16_t* x, void* ws, size_t ws_bytes, void* stream);

/* Copies bf16 rows: dst[rows_map[r]][:] = src[r][:] (dev, d_model wide), e.g. text embeddings
 * into the decoder's input sequence. */
int spd_scatter_rows(const spd_model* m, const uint16_t* src, int rows, const int32_t* rows_map,
                     uint16_t* dst, void* stream);

/* Workspace bytes of spd_attention for n_q queries in n_seqs sequences. */
size_t spd_attention_workspace_size(int n_q, int n_seqs);

/* The attention step of a decoder layer on its own (Sec. 3.2 VSkip-Attn: only the active tokens
 * are queries; every token of a sequence is a key and a value of that sequence):
 *   o_i = softmax_{t <= pos_i} (q_i . k_t / sqrt(head_dim)) v_t   per head, head h reading K/V head
 *   h / (n_heads / n_kv_heads), keys t of the query's own sequence.
 * q (dev) bf16 [n_q][n_heads * head_dim]: the queries of sequence b are rows [q_cu[b], q_cu[b+1]),
 * positions q_pos (dev int32 [n_q]) strictly ascending within a sequence and in [0, its length).
 * kv (dev) bf16 [n_kv][2 * n_kv_heads * head_dim]: per token K (rotated) then V; the tokens of
 * sequence b are rows [cu_seqlens[b], cu_seqlens[b+1]). q_cu and cu_seqlens are HOST int32 [n_seqs+1]
 * from 0 to n_q and n_kv. o (dev) bf16 [n_q][n_heads * head_dim]. head_dim 64 or 128.
 * Positions that break the precondition give wrong values, never an out-of-bounds access.
 * Errors: SPD_EINVAL, SPD_EUNSUPPORTED (head_dim), SPD_ENOSPC; device timeouts in the workspace's
 * status word. */
int spd_attention(const uint16_t* q, int n_q, const int32_t* q_pos, const int32_t* q_cu,
                  const uint16_t* kv, int n_kv, const int32_t* cu_seqlens, int n_seqs, int n_heads,
                  int n_kv_heads, int head_dim, uint16_t* o, void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes of spd_prefill for up to `max_tokens` packed tokens in up to `max_seqs` sequences. */
size_t spd_prefill_workspace_size(const spd_model* m, int max_tokens, int max_seqs);

/* Decoder prefill with per-token sub-layer bypass (Sec. 3.2 VSkip-Attn / VSkip-FFN; Alg. 1 "Forward
 * layer l, bypassing sub-layer target(i)"), LLaMA-style layers:
 *   h = x;  per layer l:  a = RMSNorm(h); K, V = RoPE(a Wk^T), a Wv^T for ALL tokens;
 *           for attention-active tokens i: h_i += Wo . Attn(RoPE(a_i Wq^T), K, V) (causal, own sequence);
 *           for FFN-active tokens i: h_i += Wdown (SiLU(Wgate b_i) * (Wup b_i)), b_i = RMSNorm(h_i).
 *   A token whose mask bit is set at layer l is not a query there (bit 0) and/or skips the FFN
 *   (bit 1): its residual row passes through that sub-layer bit-exactly; with bit 0 it still serves
 *   as a key and a value. Sub-layers with no active token launch nothing.
 *   logits[b] = lm_head . RMSNorm(h[last token of sequence b]).
 * x (dev) bf16 [n_tokens][d_model]: packed sequences; cu_seqlens (host) int32 [n_seqs + 1],
 * increasing from 0 to n_tokens; positions restart at 0 in every sequence.
 * skip_mask (host) uint8 [n_layers][n_tokens] (spd_plan_* produce it); NULL = no skipping.
 * h (dev) fp32 [n_tokens][d_model]: receives the final residual stream.
 * logits (dev, may be NULL) fp32 [n_seqs][vocab].
 * Returns once all work is enqueued. Errors: SPD_EINVAL, SPD_ENOSPC, SPD_ECUDA. */
int spd_prefill(const spd_model* m, const uint16_t* x, int n_tokens, const int32_t* cu_seqlens,
                int n_seqs, const uint8_t* skip_mask, float* h, float* logits, void* ws,
                size_t ws_bytes, void* stream);

/* ASL-Skip's online plan (Sec. 4.2, Eq. 6, Alg. 1 stage 2). */
typedef struct {
  float t_skip;                /* T_skip: a token enters skip mode once its accumulated score reaches it */
  float w1, w2;                /* weights of the online score S_sa and of SLC^Norm (Eq. 6) */
  int window;                  /* decision layers 0 .. window-1 (Alg. 1: l <= L/2) */
  const float* slc_norm;       /* host [n_layers]: SLC^Norm of layer l's designated sub-layer (Eq. 5) */
  const uint8_t* layer_target; /* host [n_layers]: m(l), 1 = attention, 2 = FFN */
  const uint8_t* is_visual;    /* host [n_tokens]: 1 for the visual tokens (the skip candidates) */
  int ablate;                  /* bit set of SPD_SKIP_NO_* below; 0 = the method as printed */
  int device_plan;             /* 0: each window layer's admissions are read back to the host, which
                                  builds that layer's row lists (one stream synchronisation per
                                  window layer; sub-layers without active tokens launch nothing).
                                  1: admissions and row lists stay on the device (a list-building
                                  kernel per window layer; the sub-layers run over every row with
                                  the lists' padding skipped); one synchronisation at the end. */
} spd_skip_policy;

/* Ablation variants of ASL-Skip (the ASL-Skip ablation table). w1 = 0 is the variant without
 * S_sa (every visual token follows the offline SLC list; no logit lens runs).
 *   SPD_SKIP_NO_ENTROPY  S_sa = ReLU(1 - F_itc) (no logit lens runs)
 *   SPD_SKIP_NO_ITC      S_sa = ReLU(1 - E_ii)
 *   SPD_SKIP_NO_ACCUM    S_skip(i) = w1 S_sa + w2 SLC^Norm(l) of the current layer only
 *   SPD_SKIP_NO_SLC      no SLC^Norm term, and an admitted token bypasses both sub-layers from its
 *                        admission layer on (whole layers instead of m(l)) */
#define SPD_SKIP_NO_ENTROPY 1
#define SPD_SKIP_NO_ITC 2
#define SPD_SKIP_NO_ACCUM 4
#define SPD_SKIP_NO_SLC 8

/* Workspace bytes of spd_prefill_adaptive for up to `max_tokens` tokens in `max_seqs` sequences. */
size_t spd_prefill_adaptive_workspace_size(const spd_model* m, int max_tokens, int max_seqs);

/* spd_prefill with the skip plan computed online instead of given. Before each layer l < window,
 * every visual token i not yet in skip mode gets
 *   E_ii  = entropy of softmax(W_unembed . RMSNorm_final(h_i)) / log V (the logit-lens reading),
 *   F_itc = (cos(h_i, q_t) + 1) / 2, q_t the mean hidden state of the text tokens of i's sequence
 *           (F_itc = 1/2 when it has none),
 *   S_sa  = ReLU(1 - E_ii - F_itc),  S_skip(i) += w1 S_sa + w2 SLC^Norm(l),
 * and enters skip mode when S_skip(i) >= T_skip, bypassing sub-layer m(l) (frozen) from layer l
 * on. Arguments as spd_prefill; admit_layer (HOST int16 [n_tokens]) receives each token's
 * admission layer (-1 = never); the call returns once it is filled (see device_plan for where the
 * decisions are taken). device_plan = 1 supports at most 1024 sequences.
 * Errors as spd_prefill. */
int spd_prefill_adaptive(const spd_model* m, const uint16_t* x, int n_tokens, const int32_t* cu_seqlens,
                         int n_seqs, const spd_skip_policy* policy, int16_t* admit_layer, float* h,
                         float* logits, void* ws, size_t ws_bytes, void* stream);

/* Bytes of a KV cache for n_seqs sequences of up to max_len tokens: per layer l, per sequence b,
 * per position p, the row [K (rotated) | V] bf16 of 2 * n_kv_heads * head_dim values, at row
 * (l * n_seqs + b) * max_len + p. The caller allocates it ZERO-FILLED: the attention reads key
 * blocks past a sequence's length with zero weight, and unwritten rows must hold finite values. */
size_t spd_kv_cache_bytes(const spd_model* m, int n_seqs, int max_len);

/* spd_prefill that also leaves every layer's K and V of every token in kv_cache (sequence b's
 * position p -> row b * max_len + p of each layer's block), for later decode steps. Tokens that
 * bypass attention at a layer still write their K and V (they are keys and values of the others).
 * The workspace is spd_prefill's. Errors as spd_prefill; SPD_EINVAL if a sequence exceeds max_len. */
int spd_prefill_kv(const spd_model* m, const uint16_t* x, int n_tokens, const int32_t* cu_seqlens,
                   int n_seqs, const uint8_t* skip_mask, float* h, float* logits, uint16_t* kv_cache,
                   int max_len, void* ws, size_t ws_bytes, void* stream);

/* Workspace bytes of spd_decode for n_seqs sequences. */
size_t spd_decode_workspace_size(const spd_model* m, int n_seqs);

/* One generation step after spd_prefill_kv: x (dev bf16 [n_seqs][d_model]) holds the embedding of
 * each sequence's next token, at position pos[b] (HOST int32 [n_seqs], in [0, max_len)). Every
 * layer appends the token's K and V to the cache and attends over positions 0..pos[b] of its
 * sequence; a generated token is a text token and runs every sub-layer (the visual tokens' skip
 * targets were applied when their cache rows were written). logits (dev fp32 [n_seqs][vocab]).
 * Errors: SPD_EINVAL, SPD_ENOSPC, SPD_ECUDA. */
int spd_decode(const spd_model* m, const uint16_t* x, int n_seqs, const int32_t* pos,
               uint16_t* kv_cache, int max_len, float* logits, void* ws, size_t ws_bytes,
               void* stream);

/* ------------------------------------------------------------------------------------------ */
/* Single kernels, exposed for composition and per-kernel tests                                 */
/* ------------------------------------------------------------------------------------------ */

/* Epilogues of spd_linear. All but SPD_EPI_ADD_F32 give bit-identical results run to run; the
 * residual update adds with fire-and-forget atomics, so where K is split across CTAs the fp32
 * additions land in no fixed order (results agree to rounding). */
typedef enum {
  SPD_EPI_F32 = 0,       /* out fp32 [M][N] = acc */
  SPD_EPI_BF16 = 1,      /* out bf16 [M][N] = bf16(acc) */
  SPD_EPI_BIAS_BF16 = 2, /* out bf16 = bf16(acc + bias[n]) */
  SPD_EPI_BIAS_GELU_BF16 = 3, /* out bf16 = bf16(GELU(acc + bias[n])) */
  SPD_EPI_ADD_F32 = 4    /* out fp32 [rows[m]][n] += acc (residual update; rows may be NULL = m) */
} spd_epilogue;

/* Workspace bytes of spd_linear for an M x N output. */
size_t spd_linear_workspace_size(int M, int N);

/* out = epilogue(X W^T) on the tcgen05 tensor cores, fp32 accumulation.
 * X (dev) bf16 [M][K]; W (dev) bf16 [N][K]; K a multiple of 8; N a multiple of 128 (or equal to
 * a padded weight count whose extra rows are never written); bias (dev) bf16 [N] or NULL; rows (dev)
 * int32 [M] or NULL; out (dev) as described by the epilogue, row stride ldo elements. */
int spd_linear(const uint16_t* X, int M, int K, const uint16_t* W, int N, int epilogue,
               const uint16_t* bias, const int32_t* rows, void* out, int ldo, void* ws,
               size_t ws_bytes, void* stream);

/* Capacity of the scratch that spd_linear_noalloc keeps inside the library. */
#define SPD_LINEAR_NOALLOC_SCRATCH_BYTES (8u << 20) /* 8 MiB of device memory */
#define SPD_LINEAR_NOALLOC_MAX_TILES 4096           /* tile counters: 2 ceil(N / 256) x ceil(M / 256) */

/* spd_linear without a workspace argument. The paper has no counterpart: this is a convenience of
 * the library, for callers that have no device buffer to lend at the point of the call and must
 * not allocate one there - e.g. a plain C host without a device memory pool, or a latency-bound
 * loop where cudaMalloc would stall the device and its memory budget is already handed out.
 * Same operation, arguments, layouts and results as spd_linear (within the same rounding: the
 * partial-sum scratch is smaller, so a large problem may be split over fewer CTAs).
 * Its scratch is one file-scope device array of SPD_LINEAR_NOALLOC_SCRATCH_BYTES in this library,
 * shared by all callers of a device: calls that may overlap on the GPU (other streams, other host
 * threads) race on it and must be serialized by the caller. The call allocates and frees nothing:
 * it clears the scratch's status word and tile counters on `stream`, then launches the GEMM.
 * The first call on a device (the device current at the call) looks up the scratch's address on
 * that device (cudaGetSymbolAddress) and caches it; make that first call before any stream capture.
 * status (dev, may be NULL): int32 receiving this call's device-side status (0 = OK, else an
 * spd_status, e.g. SPD_ETIMEOUT) once the work completes. With NULL a device-side failure of the
 * call is not reported anywhere: the scratch's own status word is cleared by the next call and no
 * entry point reads it.
 * Errors: SPD_EINVAL; SPD_ENOSPC when the problem needs more than SPD_LINEAR_NOALLOC_MAX_TILES tile
 * counters, counted as 2 ceil(N / 256) x ceil(M / 256) (the most any tiling of the GEMM uses;
 * detected on the host before anything is enqueued); SPD_ECUDA. */
int spd_linear_noalloc(const uint16_t* X, int M, int K, const uint16_t* W, int N, int epilogue,
                       const uint16_t* bias, const int32_t* rows, void* out, int ldo, int* status,
                       void* stream);

/* ------------------------------------------------------------------------------------------ */
/* One whole step (Alg. 1: stage 1 then stage 2) in one call                                    */
/* ------------------------------------------------------------------------------------------ */

/* Workspace bytes of spd_step for this model, pruning configuration and batch layout (0 on
 * invalid arguments). */
size_t spd_step_workspace_size(const spd_model* m, const spd_prune_cfg* cfg, int n_seqs,
                               const int32_t* tiles_per_seq, const int32_t* text_len);

/* The whole SPIDER prefill of a batch (Alg. 1): MSV-Prune of every tile (spd_prune), the kept
 * final-layer rows to bf16 (spd_gather_rows_bf16), the projector (spd_project; a row copy when the
 * model has none), the text embeddings, and the decoder prefill with the skip mask (spd_prefill).
 * Request b owns tiles_per_seq[b] consecutive tiles (host int32 [n_seqs], summing to cfg->n_tiles)
 * and text_len[b] text tokens (host int32 [n_seqs]); its sequence is [cfg->keep kept tokens of each
 * of its tiles, in tile order; its text tokens].
 * feats[l], attn, text and logits may each be in host memory (pinned or pageable) or in device
 * memory: host inputs are copied into the workspace on `stream` first and host logits are copied
 * back at the end (the caller synchronises `stream` before reading them). Layouts: feats[l] fp32
 * [n_tiles][n_tok][d_feat]; attn fp32 as in spd_prune; text bf16 [sum(text_len)][d_model], the
 * requests' text rows in request order; skip_mask (host) uint8 [n_layers][T] over the packed
 * tokens (NULL = no skipping); logits fp32 [n_seqs][vocab].
 * Errors: SPD_EINVAL, SPD_ENOSPC, SPD_ECUDA; device-side failures through spd_step_status. */
int spd_step(const spd_model* m, const spd_prune_cfg* cfg, int n_seqs, const int32_t* tiles_per_seq,
             const int32_t* text_len, const float* const* feats, const float* attn, const uint16_t* text,
             const uint8_t* skip_mask, float* logits, void* ws, size_t ws_bytes, void* stream);

/* The first device-side failure recorded by the calls of a spd_step workspace (synchronises
 * `stream`, clears the status words): SPD_OK or a negative spd_status. */
int spd_step_status(void* ws, const spd_model* m, const spd_prune_cfg* cfg, int n_seqs,
                    const int32_t* tiles_per_seq, const int32_t* text_len, void* stream);

/* ------------------------------------------------------------------------------------------ */
/* The hot path's contract names (thin forms of the calls above)                               */
/* ------------------------------------------------------------------------------------------ */

/* = spd_prune_workspace_size. */
size_t spd_prune_workspace(const spd_prune_cfg* cfg);

/* = spd_prefill_workspace_size. */
size_t spd_prefill_workspace(const spd_model* m, int total_tokens, int n_seqs);

/* = spd_gather_rows_bf16 with the kept patch indices of spd_prune: out[t * keep + j][:] =
 * bf16(payload[t][has_cls + keep_idx[t][j]][:]). payload (dev) fp32 [n_tiles][n_tok][d] (n_tok rows
 * per tile, including the [CLS] row when has_cls); keep_idx (dev) int32 [n_tiles][keep]; out (dev)
 * bf16 [n_tiles * keep][d]; d a multiple of 4. Out-of-range indices are skipped (no report).
 * Errors as spd_gather_rows_bf16. */
int spd_gather_bf16(const float* payload, int n_tok, const int32_t* keep_idx, int n_tiles, int keep,
                    int has_cls, int d, uint16_t* out, void* stream);

/* Copies the message of the calling thread's last failed call (spd_last_error) into buf, at most
 * n - 1 characters and a terminating NUL (n > 0). Returns the message's full length. */
int spd_last_error_detail(char* buf, size_t n);

/* Device-side status of a workspace (synchronises `stream`): SPD_OK or the first failure recorded
 * since the last read (which it clears), or a negative status of the read itself. */
int spd_check(void* ws, void* stream);

/* = spd_plan_static: a per-layer mask applied to the selected (visual) tokens. */
int spd_plan_from_layer_mask(int n_layers, int n_tokens, const uint8_t* layer_mask,
                             const uint8_t* token_is_visual, uint8_t* mask);

/* spd_prefill with Alg. 1's plan in its per-token form: token i bypasses target[i] (1 attention,
 * 2 FFN, 3 both) in every layer l >= admit_layer[i] (-1 = never). admit_layer (HOST int16
 * [n_tokens]) and target (HOST uint8 [n_tokens]) are expanded on the host (spd_plan_adaptive);
 * both NULL = no skipping. Other arguments and errors as spd_prefill. */
int spd_prefill_admit(const spd_model* m, const uint16_t* x, int n_tokens, const int32_t* cu_seqlens,
                      int n_seqs, const int16_t* admit_layer, const uint8_t* target, float* h,
                      float* logits, void* ws, size_t ws_bytes, void* stream);

#ifdef __cplusplus
}
#endif
#endif /* SPIDER_H */
