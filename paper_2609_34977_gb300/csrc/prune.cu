// MSV-Prune (Sec. 4.1, Eq. 1-3; Alg. 1 stage 1) on the GPU, every tile independently.
//
//   rowstats     a_v = head-mean of the attention (Sec. 4.1.1); 1/||F_l,i|| for every tapped layer
//                (and ||F_l,i||^2, or the log-sum-exp and negentropy of softmax(F_l,i), for the
//                MSE and KL ablations of sim)
//   anchors      top-N_anc of a_v by ranking (a_v desc, index asc) keys (Eq. 1); stable lists of
//                anchor and non-anchor tokens by block prefix sums
//   anchor_sim   a_i = max_p cos(F^L_i, F^L_p) over anchors: 64 x 64 register-tiled fp32 products,
//                the feature dimension split over a cluster of 4 (8 for few tiles) CTAs whose partial tiles are summed
//                in rank order through distributed shared memory; max via atomicMax on
//                order-preserving integer keys (exact, order independent)
//   kmeans       one thread-block cluster of 16 CTAs per tile, each owning a contiguous slice of the
//                non-anchor tokens whose F^L rows it keeps in shared memory for every iteration (8
//                CTAs re-reading them from L2 where they do not fit, 4 beyond one wave of such
//                clusters): Lloyd on raw F^L (assignment
//                in each CTA, per-CTA sums in token order, cross-CTA sums in rank order through
//                distributed shared memory), then the
//                per-cluster, per-layer sums of unit feature rows, the sums of a_j, sizes and Eq. 2
//                quotas
//   scores       s_i = [sum_l w_l f_i . (S_l,k - f_i)] / (|C_k| - 1) + a_i + (A_k - a_i) / (|C_k| - 1),
//                the per-token mean of Eq. 3's S_ij over the other members of its cluster (for
//                the MSE and KL ablations the same cluster-sum identity with raw rows, plus the
//                per-cluster sums of ||F_j||^2 or of the log-sum-exps)
//   select       per cluster the N_k lowest (score, index) keys; kept = anchors + selected, compacted
//                in ascending index order
// Where the rows are resident and the similarity is the cosine, the K-means kernel goes on to the
// scores and the selection itself (fused_select): four launches instead of six.
// All reductions run in a fixed order, so repeated runs give identical bits.
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include <cooperative_groups.h>

#include <algorithm>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace cg = cooperative_groups;

namespace spd {

struct PruneDims {
  int n_tiles, n_tok, off, n, d, L, fin, H, form, n_att, keep, K, iters, n_anc, n_cmp, m;
  int sim;        // SPD_SIM_*
  float wf, wa;   // weights (0 or 1) of the final-layer intra-cluster term and the anchor bracket
  float w[SPD_MAX_FEAT_LAYERS];
  const float* feat[SPD_MAX_FEAT_LAYERS];
};

struct PruneWs {
  float* a_v;       // [T][n]
  float* inv;       // [L][T][n]
  float* st1;       // [L][T][n] MSE: ||F_l,i||^2; KL: log-sum-exp of F_l,i (rounded to fp32)
  float* st2;       // [L][T][n] KL: sum_c P_c log P_c of P = softmax(F_l,i)
  float* st3;       // [L][T][n] KL: log-sum-exp minus its fp32 rounding (st1 + st3 = the fp64 value)
  int8_t* role;     // [T][n] 1 anchor
  int32_t* alist;   // [T][n_anc]
  int32_t* ulist;   // [T][m]
  uint32_t* asim;   // [T][n] ordered keys of a_i
  int32_t* assign;  // [T][m]
  int32_t* counts;  // [T][16]
  int32_t* quotas;  // [T][16]
  float* asum;      // [T][16]
  float* csum;      // [T][L][K][d]
  double* ssum;     // [T][L][16] MSE / KL: per-cluster sums of st1 (+ st3), in fp64
  float* score;     // [T][m]
  int* status;
};

// The outputs of a prune call (kind, cluster and scores optional).
struct PruneOut {
  int32_t* keep_idx;
  uint8_t* kind;
  int8_t* cluster;
  float* scores;
};

namespace {

__device__ __forceinline__ uint32_t ordered_key(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float ordered_val(uint32_t u) {
  return __uint_as_float((u & 0x80000000u) ? (u & 0x7fffffffu) : ~u);
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}
__device__ __forceinline__ double warp_sum_d(double v) {
#pragma unroll
  for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// Ascending bitonic sort of N (power of two) keys in shared memory by the whole block.
__device__ void bitonic_sort(uint64_t* keys, int N) {
  for (int k = 2; k <= N; k <<= 1) {
    for (int j = k >> 1; j > 0; j >>= 1) {
      for (int i = threadIdx.x; i < N; i += blockDim.x) {
        const int ixj = i ^ j;
        if (ixj > i) {
          const bool up = (i & k) == 0;
          const uint64_t a = keys[i], b = keys[ixj];
          if ((a > b) == up) {
            keys[i] = b;
            keys[ixj] = a;
          }
        }
      }
      __syncthreads();
    }
  }
}

// Position of every key in the ascending order of keys[0..N) (distinct keys): the number of smaller
// keys, counted by each thread for its keys (broadcast shared-memory reads, no barriers). rank_of
// is called with (i, rank) for i < N.
template <typename F>
__device__ __forceinline__ void rank_keys(const uint64_t* keys, int N, F rank_of) {
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    const uint64_t ki = keys[i];
    int r0 = 0, r1 = 0, r2 = 0, r3 = 0;
    int j = 0;
    for (; j + 4 <= N; j += 4) {
      r0 += keys[j] < ki;
      r1 += keys[j + 1] < ki;
      r2 += keys[j + 2] < ki;
      r3 += keys[j + 3] < ki;
    }
    for (; j < N; ++j) r0 += keys[j] < ki;
    rank_of(i, r0 + r1 + r2 + r3);
  }
}
constexpr int kRankMax = 2048;  // longest list ranked by counting; longer ones are sorted

// Exclusive prefix sum of one int per thread over a block of 1024 threads.
__device__ int block_scan_excl(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) tmp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = (lane < (int)(blockDim.x >> 5)) ? tmp[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, off);
      if (lane >= off) w += y;
    }
    tmp[lane] = w;  // inclusive totals of warps
  }
  __syncthreads();
  const int before = (warp ? tmp[warp - 1] : 0) + x - v;
  if (total) *total = tmp[(blockDim.x >> 5) - 1];
  __syncthreads();
  return before;
}

__device__ __forceinline__ const float* feat_row(const PruneDims& p, int l, int t, int i) {
  return p.feat[l] + (size_t(t) * p.n_tok + p.off + i) * p.d;
}

// ---- 1. a_v and inverse norms ---------------------------------------------------------------
template <int SIM>
__global__ void __launch_bounds__(256) rowstats_kernel(PruneDims p, const float* attn,
                                                       PruneWs w) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int i = blockIdx.x * 8 + warp;
  if (i >= p.n) return;
  for (int l = 0; l < p.L; ++l) {
    const float4* r = reinterpret_cast<const float4*>(feat_row(p, l, t, i));
    float ss = 0.0f;
    for (int c = lane; c < p.d / 4; c += 32) {
      const float4 v = r[c];
      ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = warp_sum(ss);
    const size_t o = (size_t(l) * p.n_tiles + t) * p.n + i;
    if (lane == 0) w.inv[o] = 1.0f / sqrtf(ss);
    if (SIM == SPD_SIM_MSE && lane == 0) w.st1[o] = ss;
    if (SIM == SPD_SIM_KL) {
      // softmax over the row in fp64 (z = x - max exact, e^z, sums): the KL scores multiply the
      // log-probabilities by log-ratios of tens, so an fp32 log-sum-exp (about 2e-6 off) would
      // move them by about 1e-4
      float mx = -INFINITY;
      for (int c = lane; c < p.d / 4; c += 32) {
        const float4 v = r[c];
        mx = fmaxf(mx, fmaxf(fmaxf(v.x, v.y), fmaxf(v.z, v.w)));
      }
#pragma unroll
      for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
      double se = 0.0, te = 0.0;
      for (int c = lane; c < p.d / 4; c += 32) {
        const float4 v = r[c];
        const double z[4] = {double(v.x) - mx, double(v.y) - mx, double(v.z) - mx, double(v.w) - mx};
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const double e = exp(z[u]);
          se += e;
          te += e * z[u];
        }
      }
      se = warp_sum_d(se);
      te = warp_sum_d(te);
      if (lane == 0) {
        const double lse = double(mx) + log(se);  // log sum_c e^x_c
        const float hi = float(lse);
        w.st1[o] = hi;
        w.st3[o] = float(lse - double(hi));
        w.st2[o] = float(te / se - log(se));      // sum_c P_c log P_c
      }
    }
  }
  if (lane == 0) {
    const int col = (p.form == 0) ? 1 + i : i;
    float s = 0.0f;
    for (int h = 0; h < p.H; ++h) s += attn[(size_t(t) * p.H + h) * p.n_att + col];
    w.a_v[size_t(t) * p.n + i] = s / float(p.H);
  }
}

// ---- 2. anchors (Eq. 1) and stable token lists ------------------------------------------------
__global__ void __launch_bounds__(1024) anchor_kernel(PruneDims p, PruneWs w) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ uint64_t keys[4096];
  __shared__ int tmp[32];
  const int t = blockIdx.x;
  int N = 1;
  while (N < p.n) N <<= 1;
  // (a_v descending, index ascending) as ascending 64-bit keys
  for (int i = threadIdx.x; i < N; i += blockDim.x) {
    uint64_t k = ~0ull;
    if (i < p.n)
      k = (uint64_t(~ordered_key(w.a_v[size_t(t) * p.n + i])) << 32) | uint32_t(i);
    keys[i] = k;
  }
  __syncthreads();
  int8_t* role = w.role + size_t(t) * p.n;
  if (p.n <= kRankMax) {
    // anchor iff its key is among the n_anc smallest
    rank_keys(keys, p.n, [&](int i, int r) { role[i] = r < p.n_anc ? 1 : 0; });
  } else {
    bitonic_sort(keys, N);
    for (int i = threadIdx.x; i < p.n; i += blockDim.x) role[i] = 0;
    __syncthreads();
    for (int r = threadIdx.x; r < p.n_anc; r += blockDim.x) role[keys[r] & 0xffffffffu] = 1;
  }
  __syncthreads();
  // stable lists: each thread owns 4 consecutive tokens
  const int base = threadIdx.x * 4;
  int na = 0;
  for (int q = 0; q < 4; ++q)
    if (base + q < p.n) na += role[base + q];
  const int nu = ((base < p.n) ? min(4, p.n - base) : 0) - na;
  const int a0 = block_scan_excl(na, tmp, nullptr);
  const int u0 = block_scan_excl(nu, tmp, nullptr);
  int ai = a0, ui = u0;
  // a_i = 0 where the anchor bracket is absent (no anchors, or the ablation without it)
  const uint32_t init = (p.n_anc == 0 || p.wa == 0.0f) ? ordered_key(0.0f) : 0u;
  for (int q = 0; q < 4; ++q) {
    const int i = base + q;
    if (i >= p.n) break;
    if (role[i]) w.alist[size_t(t) * p.n_anc + ai++] = i;
    else w.ulist[size_t(t) * p.m + ui++] = i;
    w.asim[size_t(t) * p.n + i] = init;
  }
}

// ---- 3. a_i = max over anchors of cos(F^L_i, F^L_p) -------------------------------------------
// A cluster of AS CTAs per 64 non-anchor tokens x 64 anchors tile, each CTA one slice of the
// feature dimension: 32-wide chunks through shared memory (stored transposed; the next chunk is
// fetched into registers while the current one is multiplied), 4 x 4 dot products per thread
// (4 consecutive rows x 4 consecutive anchors: two 16-byte shared-memory loads per 16 FMAs).
// The partial tiles are summed in rank order through distributed shared memory, each CTA
// finishing 64 / AS rows. AS = 4 at serving batch; 8 for a few tiles (shorter chains per CTA).
template <int SIM, int AS>
__global__ void __cluster_dims__(AS, 1, 1) __launch_bounds__(256)
    anchor_sim_kernel(PruneDims p, PruneWs w) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ __align__(16) float Us[32][68], As[32][68];
  __shared__ float P[64][65];  // this CTA's partial dot products
  cg::cluster_group cl = cg::this_cluster();
  const int rank = int(cl.block_rank());
  const int t = blockIdx.z, tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int u0 = (blockIdx.x / AS) * 64, p0 = blockIdx.y * 64;
  const int* ul = w.ulist + size_t(t) * p.m;
  const int* al = w.alist + size_t(t) * p.n_anc;
  // staging: thread loads column dd of rows 8 r0 + i (i < 8) of both operands
  const int dd = threadIdx.x & 31, r0 = threadIdx.x >> 5;
  // per-row statistics of the final layer (MSE: squared norms; KL: log-sum-exps, negentropies)
  const size_t so = (size_t(p.fin) * p.n_tiles + t) * p.n;
  constexpr bool kl = SIM == SPD_SIM_KL;
  // rows as 32-bit offsets into the tile's block of F^L (fewer registers than pointers; the block
  // holds at most 4097 rows of at most 4096 floats); -1 for rows past the lists
  const float* tile_f = feat_row(p, p.fin, t, -p.off);
  int uo[8], ao[8];
  double ulse[8];  // KL: the non-anchor operand is softmax(F^L_i) = exp(F^L_i - lse_i), in fp64
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const int r = 8 * r0 + i;
    const bool uv = u0 + r < p.m;
    uo[i] = uv ? (p.off + ul[u0 + r]) * p.d : -1;
    ao[i] = (p0 + r < p.n_anc) ? (p.off + al[p0 + r]) * p.d : -1;
    ulse[i] = (kl && uv) ? double(w.st1[so + ul[u0 + r]]) + double(w.st3[so + ul[u0 + r]]) : 0.0;
  }
  const int nch = (p.d + 31) / 32, c0 = rank * nch / AS, c1 = (rank + 1) * nch / AS;
  float ru[8], ra[8];
  auto fetch = [&](int ch) {
    const int dcol = ch * 32 + dd;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const float x = (uo[i] >= 0 && dcol < p.d) ? tile_f[uo[i] + dcol] : 0.0f;
      if constexpr (kl) ru[i] = (uo[i] >= 0 && dcol < p.d) ? float(exp(double(x) - ulse[i])) : 0.0f;
      else ru[i] = x;
      ra[i] = (ao[i] >= 0 && dcol < p.d) ? tile_f[ao[i] + dcol] : 0.0f;
    }
  };
  float acc[4][4];
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
  if (c0 < c1) fetch(c0);
  for (int ch = c0; ch < c1; ++ch) {
    // eight consecutive rows of column dd: two 16-byte stores per operand
    *reinterpret_cast<float4*>(&Us[dd][8 * r0]) = make_float4(ru[0], ru[1], ru[2], ru[3]);
    *reinterpret_cast<float4*>(&Us[dd][8 * r0 + 4]) = make_float4(ru[4], ru[5], ru[6], ru[7]);
    *reinterpret_cast<float4*>(&As[dd][8 * r0]) = make_float4(ra[0], ra[1], ra[2], ra[3]);
    *reinterpret_cast<float4*>(&As[dd][8 * r0 + 4]) = make_float4(ra[4], ra[5], ra[6], ra[7]);
    __syncthreads();
    if (ch + 1 < c1) fetch(ch + 1);  // in flight during the products below
#pragma unroll 8
    for (int e = 0; e < 32; ++e) {
      // rows 4 ty .. 4 ty + 3 and anchors 4 tx .. 4 tx + 3: one 16-byte load each
      const float4 av = *reinterpret_cast<const float4*>(&Us[e][4 * ty]);
      const float4 bv = *reinterpret_cast<const float4*>(&As[e][4 * tx]);
      const float a[4] = {av.x, av.y, av.z, av.w}, b[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] += a[i] * b[j];
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) P[4 * ty + i][4 * tx + j] = acc[i][j];
  cl.sync();
  // rows RPC rank .. RPC rank + RPC - 1 of the tile (TPR threads a row, CPT columns a thread): all
  // AS partials loaded first, summed in rank order
  constexpr int RPC = 64 / AS, TPR = 256 / RPC, CPT = 64 / TPR;
  const int lr = RPC * rank + int(threadIdx.x) / TPR, cx = int(threadIdx.x) % TPR;
  float x[AS][CPT];
#pragma unroll
  for (int src = 0; src < AS; ++src) {
    const float* pp = cl.map_shared_rank(&P[0][0], src) + lr * 65;
#pragma unroll
    for (int j = 0; j < CPT; ++j) x[src][j] = pp[cx + TPR * j];
  }
  const float* inv = w.inv + size_t(p.fin) * p.n_tiles * p.n + size_t(t) * p.n;
  const int ur = u0 + lr;
  float best = -INFINITY;
  // candidates whose maximum over p gives a_i through an increasing map g:
  //   cos: F_i.F_p / (|F_i| |F_p|)             (g = identity)
  //   MSE: 2 F_i.F_p - |F_p|^2                  (g(v) = -(|F_i|^2 - v) / d)
  //   KL:  P_i.F_p - lse_p = -KL(P_i||P_p) + N_i (g(v) = v - N_i)
  if (ur < p.m) {
    const float iu = inv[ul[ur]];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
      float sdot = 0.0f;
#pragma unroll
      for (int src = 0; src < AS; ++src) sdot += x[src][j];
      const int pa = p0 + cx + TPR * j;
      if (pa < p.n_anc) {
        const int ia = al[pa];
        const float v = SIM == SPD_SIM_COS ? sdot * iu * inv[ia]
                        : SIM == SPD_SIM_MSE ? 2.0f * sdot - w.st1[so + ia]
                                             : float(double(sdot) - double(w.st1[so + ia]) -
                                                     double(w.st3[so + ia]));
        best = fmaxf(best, v);
      }
    }
  }
#pragma unroll
  for (int off = TPR / 2; off; off >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, off));
  if (cx == 0 && ur < p.m) {
    const int iu = ul[ur];
    if (SIM == SPD_SIM_MSE) best = -(w.st1[so + iu] - best) / float(p.d);
    else if (SIM == SPD_SIM_KL) best = best - w.st2[so + iu];
    atomicMax(&w.asim[size_t(t) * p.n + iu], ordered_key(best));
  }
  cl.sync();  // peers read this CTA's partial tile above
}

// ---- 4. K-means (Lloyd) and Eq. 2 quotas ------------------------------------------------------
__device__ void compute_quotas(const int* sizes, int K, int n_cmp, int* quota) {
  int total = 0, nonempty = 0;
  for (int k = 0; k < K; ++k) {
    quota[k] = 0;
    total += sizes[k];
    nonempty += sizes[k] > 0;
  }
  if (n_cmp <= 0 || total == 0) return;
  int order[SPD_MAX_CLUSTERS];
  if (n_cmp < nonempty) {  // one each to the largest clusters, ties to the lower k
    for (int k = 0; k < K; ++k) order[k] = k;
    for (int a = 1; a < K; ++a)
      for (int b = a; b > 0 && (sizes[order[b]] > sizes[order[b - 1]]); --b) {
        const int x = order[b]; order[b] = order[b - 1]; order[b - 1] = x;
      }
    for (int r = 0; r < n_cmp; ++r) quota[order[r]] = 1;
    return;
  }
  long long rem[SPD_MAX_CLUSTERS];
  int sum = 0;
  for (int k = 0; k < K; ++k) {
    const long long num = (long long)n_cmp * sizes[k];
    rem[k] = num % total;
    if (sizes[k] > 0) {
      int q = int((2 * num + total) / (2LL * total));  // round half away from zero
      if (q < 1) q = 1;
      if (q > sizes[k]) q = sizes[k];
      quota[k] = q;
    }
    sum += quota[k];
  }
  if (sum < n_cmp) {  // descending fractional part, ties to the lower k
    for (int k = 0; k < K; ++k) order[k] = k;
    for (int a = 1; a < K; ++a)
      for (int b = a; b > 0 && rem[order[b]] > rem[order[b - 1]]; --b) {
        const int x = order[b]; order[b] = order[b - 1]; order[b - 1] = x;
      }
    while (sum < n_cmp)
      for (int r = 0; r < K && sum < n_cmp; ++r)
        if (quota[order[r]] < sizes[order[r]]) { ++quota[order[r]]; ++sum; }
  } else if (sum > n_cmp) {  // ascending fractional part, ties to the higher k
    for (int k = 0; k < K; ++k) order[k] = K - 1 - k;
    for (int a = 1; a < K; ++a)
      for (int b = a; b > 0 && rem[order[b]] < rem[order[b - 1]]; --b) {
        const int x = order[b]; order[b] = order[b - 1]; order[b - 1] = x;
      }
    while (sum > n_cmp)
      for (int r = 0; r < K && sum > n_cmp; ++r)
        if (quota[order[r]] > 1) { --quota[order[r]]; --sum; }
  }
}

// The fused tail of the K-means kernel: every CTA turns its tokens' accumulated terms into Eq. 3
// scores (as score_kernel) and pushes their (cluster, score, index) keys into every CTA; each CTA
// ranks its own tokens among all non-anchor keys and marks the selected ones in CTA 0, which
// compacts the kept tokens in index order (as select_kernel). keys: 8 (m + 1) + n bytes of every
// CTA's shared memory that nothing else reads any more (the resident rows); j0: this CTA's first
// token of the tile's non-anchor list.
template <int KC>
__device__ void fused_select(const PruneDims& p, const PruneWs& w, const PruneOut& out,
                             cg::cluster_group& cl, int rank, int t, int j0, int nl,
                             const int8_t* asg, const int* idx, const float* av, float* sacc,
                             const int* ncl, const float* ak, uint64_t* keys) {
  const int m = p.m, K = p.K;
  __shared__ int seg[SPD_MAX_CLUSTERS + 1];
  __shared__ int quota[SPD_MAX_CLUSTERS];
  __shared__ int tmp[32];
  uint8_t* kept = reinterpret_cast<uint8_t*>(keys + m + 1);  // CTA 0: [n]
  __syncthreads();  // every warp's terms of the last layer are in sacc
  if (threadIdx.x == 0) {  // every CTA: segment offsets and the Eq. 2 quotas (same in all)
    int sizes[SPD_MAX_CLUSTERS], q[SPD_MAX_CLUSTERS];
    int acc = 0;
    for (int k = 0; k < K; ++k) {
      seg[k] = acc;
      sizes[k] = ncl[k];
      acc += ncl[k];
    }
    seg[K] = acc;
    compute_quotas(sizes, K, p.n_cmp, q);
    for (int k = 0; k < K; ++k) quota[k] = q[k];
  }
  uint64_t key[2];  // this thread's tokens jj = threadIdx.x + u blockDim.x (nl <= 2 blockDim.x)
  for (int u = 0; u < 2; ++u) {
    const int jj = threadIdx.x + u * blockDim.x;
    key[u] = ~0ull;
    if (jj < nl) {
      const int k = asg[jj], cnt = ncl[k];
      const float ai = av[jj];
      float s;
      if (cnt <= 1) {
        s = p.wa * 2.0f * ai;
      } else {
        const float inv_c = 1.0f / float(cnt - 1);
        s = sacc[jj] * inv_c + p.wa * (ai + (ak[k] - ai) * inv_c);
      }
      key[u] = (uint64_t(k) << 45) | (uint64_t(ordered_key(s)) << 13) | uint64_t(idx[jj]);
    }
  }
  cl.sync();  // no CTA reads its resident rows any more
  for (int u = 0; u < 2; ++u) {
    const int jj = threadIdx.x + u * blockDim.x;
    if (jj < nl)
      for (int rr = 0; rr < KC; ++rr) cl.map_shared_rank(keys, rr)[j0 + jj] = key[u];
  }
  if (rank == 0)
    for (int i = threadIdx.x; i < p.n; i += blockDim.x) kept[i] = uint8_t(w.role[size_t(t) * p.n + i]);
  cl.sync();  // every CTA holds all m keys; CTA 0 the anchor flags
  uint8_t* kept0 = cl.map_shared_rank(kept, 0);
  for (int u = 0; u < 2; ++u) {
    const int jj = threadIdx.x + u * blockDim.x;
    if (jj >= nl) continue;
    const uint64_t ki = key[u];
    int r0 = 0, r1 = 0, r2 = 0, r3 = 0, j = 0;
    for (; j + 4 <= m; j += 4) {
      r0 += keys[j] < ki;
      r1 += keys[j + 1] < ki;
      r2 += keys[j + 2] < ki;
      r3 += keys[j + 3] < ki;
    }
    for (; j < m; ++j) r0 += keys[j] < ki;
    const int k = int(ki >> 45);
    // the key at sorted position r of cluster k's segment is kept iff r - seg[k] < quota[k]
    if (r0 + r1 + r2 + r3 - seg[k] < quota[k]) kept0[ki & 0x1fffu] = 2;
    if (out.cluster) out.cluster[size_t(t) * p.n + (ki & 0x1fffu)] = int8_t(k);
    if (out.scores) out.scores[size_t(t) * p.n + (ki & 0x1fffu)] = ordered_val(uint32_t(ki >> 13));
  }
  cl.sync();  // the selected flags are in CTA 0
  if (rank != 0) return;
  // compaction in index order: thread th owns tokens [th q, th q + q)
  const int q = (p.n + blockDim.x - 1) / blockDim.x, base = threadIdx.x * q;
  int nk = 0;
  for (int u = 0; u < q; ++u)
    if (base + u < p.n) nk += kept[base + u] != 0;
  int pos = block_scan_excl(nk, tmp, nullptr);
  for (int u = 0; u < q; ++u) {
    const int i = base + u;
    if (i >= p.n) break;
    if (kept[i]) {
      if (pos < p.keep) out.keep_idx[size_t(t) * p.keep + pos] = i;
      else set_status(w.status, SPD_EINVAL);
      ++pos;
    }
    if (out.kind) out.kind[size_t(t) * p.n + i] = kept[i];
    if (kept[i] == 1) {
      if (out.cluster) out.cluster[size_t(t) * p.n + i] = -1;
      if (out.scores) out.scores[size_t(t) * p.n + i] = INFINITY;
    }
  }
}

// Row jj of this CTA's tokens: resident in shared memory (rows + jj D) or in global memory
// (g + (row0 + idx[jj]) D), optionally scaled by scale[jj].
struct RowAccess {
  const float* rows;  // resident rows, or null
  const float* g;
  size_t row0;
  const int* idx;
  int D;
  const float* scale;  // or null
  __device__ __forceinline__ const float* row(int jj) const {
    return rows ? rows + size_t(jj) * D : g + (row0 + idx[jj]) * D;
  }
  __device__ __forceinline__ float operator()(int jj, int c) const {
    const float v = row(jj)[c];
    return scale ? v * scale[jj] : v;
  }
  __device__ __forceinline__ float4 v4(int jj, int c) const {
    float4 v = *reinterpret_cast<const float4*>(row(jj) + c);
    if (scale) {
      const float sc = scale[jj];
      v.x *= sc;
      v.y *= sc;
      v.z *= sc;
      v.w *= sc;
    }
    return v;
  }
};

// part[k][c] = sum over this CTA's tokens jj of cluster k, in token order, of value(jj, c): one
// thread per column, KN accumulators in registers, eight values in flight.
template <int KN, typename F>
__device__ __forceinline__ void column_sums(float* part, int K, int D, int nl, const int8_t* asg,
                                            F value) {
  if constexpr (KN == 4) {
    // four adjacent columns per thread (float4), same token-order sums per column
    for (int c = 4 * threadIdx.x; c < D; c += 4 * blockDim.x) {
      float4 acc[KN];
#pragma unroll
      for (int k = 0; k < KN; ++k) acc[k] = make_float4(0.f, 0.f, 0.f, 0.f);
      for (int jb = 0; jb < nl; jb += 8) {
        float4 xv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u)
          xv[u] = jb + u < nl ? value.v4(jb + u, c) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (jb + u < nl) {
            const int a = asg[jb + u];
#pragma unroll
            for (int k = 0; k < KN; ++k)
              if (k == a) {
                acc[k].x += xv[u].x;
                acc[k].y += xv[u].y;
                acc[k].z += xv[u].z;
                acc[k].w += xv[u].w;
              }
          }
      }
#pragma unroll
      for (int k = 0; k < KN; ++k)
        if (k < K) *reinterpret_cast<float4*>(part + k * D + c) = acc[k];
    }
  } else {
    for (int c = threadIdx.x; c < D; c += blockDim.x) {
      float acc[KN];
#pragma unroll
      for (int k = 0; k < KN; ++k) acc[k] = 0.0f;
      for (int jb = 0; jb < nl; jb += 8) {
        float xv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) xv[u] = jb + u < nl ? value(jb + u, c) : 0.0f;
#pragma unroll
        for (int u = 0; u < 8; ++u)
          if (jb + u < nl) {
            const int a = asg[jb + u];
#pragma unroll
            for (int k = 0; k < KN; ++k)
              if (k == a) acc[k] += xv[u];
          }
      }
#pragma unroll
      for (int k = 0; k < KN; ++k)
        if (k < K) part[k * D + c] = acc[k];
    }
  }
}

// Sums over the KC CTAs of the cluster, in rank order, of the per-CTA column sums `part` (K x D in
// every CTA's shared memory), for this CTA's slice of columns; `emit(k, c, value)` consumes them.
template <int KC, typename F>
__device__ __forceinline__ void cluster_column_reduce(cg::cluster_group& cl, float* part, int K, int D,
                                                      int rank, F emit) {
  const int c0 = rank * D / KC, c1 = (rank + 1) * D / KC, width = c1 - c0;
  for (int e = threadIdx.x; e < K * width; e += blockDim.x) {
    const int k = e / width, c = c0 + e % width;
    float x[KC];
#pragma unroll
    for (int rr = 0; rr < KC; ++rr) x[rr] = cl.map_shared_rank(part, rr)[k * D + c];  // in flight
    float sum = 0.0f;
#pragma unroll
    for (int rr = 0; rr < KC; ++rr) sum += x[rr];
    emit(k, c, sum);
  }
}

// K-means over one tile per cluster of KC CTAs, CTA r owning the non-anchor tokens
// [r m / KC, (r+1) m / KC). RES: those tokens' F^L rows are copied into the CTA's shared memory
// once (one bulk copy per row) and every Lloyd iteration reads them there; otherwise each
// iteration re-reads them from global memory (L2). KN: an upper bound of K known at compile time
// (K itself for the paper's K = 4), sizing the per-thread accumulators.
template <int KN>
constexpr int kmeans_threads() { return KN == 4 ? 256 : 512; }

// COS: the similarity kind is the cosine (the paper's); the MSE / KL ablations' extra sums are
// compiled into the other instance only (the Lloyd loop is instruction-bound).
// FUSED (RES and COS only): the kernel goes on to the Eq. 3 scores of its tokens, from the resident
// rows of each layer and that layer's cluster sums pushed into every CTA, and the rank-0 CTA then
// selects and compacts the kept tokens (the work of score_kernel and select_kernel, without their
// launches and without reading the features again).
template <int KC, bool RES, int KN, bool COS, bool FUSED = false>
__global__ void __launch_bounds__(kmeans_threads<KN>()) kmeans_kernel(PruneDims p, PruneWs w,
                                                                       PruneOut out) {
  static_assert(!FUSED || (RES && COS), "the fused tail reads resident rows of unit-norm scores");
  pdl_launch_dependents();
  pdl_wait();
  extern __shared__ __align__(16) float ksm[];
  const int K = p.K, D = p.d, m = p.m;
  const int nl_max = (m + KC - 1) / KC;
  float* rows = ksm;                                          // RES: [nl_max][D]
  float* cent = ksm + (RES ? size_t(nl_max) * D : size_t(0));  // [K][D] centroids (every CTA)
  float* part = cent + size_t(K) * D;                         // [K][D] this CTA's column sums
  __shared__ int cnt[SPD_MAX_CLUSTERS];   // this CTA's cluster sizes
  __shared__ float asum_part[SPD_MAX_CLUSTERS];
  __shared__ double ssum_part[SPD_MAX_CLUSTERS];  // MSE / KL: this CTA's sums of st1 (+ st3) per cluster
  __shared__ int changed;      // this CTA's assignment changed in the current iteration
  __shared__ int any_changed;  // ... some CTA's of the cluster
  __shared__ int8_t asg[4096 / KC + 1];
  __shared__ int idx[4096 / KC + 1];     // patch index of each of this CTA's tokens
  __shared__ float av[4096 / KC + 1];    // their a_j
  __shared__ float rinv[4096 / KC + 1];  // their 1 / ||F_l,j|| (cos) or st1 (MSE, KL) of the layer
  __shared__ int ncl[SPD_MAX_CLUSTERS];  // cluster sizes over the whole cluster of CTAs
  __shared__ float ak[SPD_MAX_CLUSTERS];  // FUSED: the cluster's sums of a_j (rank order)
  __shared__ float sacc[FUSED ? 4096 / KC + 1 : 1];  // FUSED: per token, sum_l w_l f_i.(S_l,k - f_i)
  __shared__ uint64_t rows_bar;
  cg::cluster_group cl = cg::this_cluster();
  const int rank = int(cl.block_rank());
  const int t = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nw = blockDim.x >> 5;
  const int j0 = rank * m / KC, j1 = (rank + 1) * m / KC, nl = j1 - j0;
  const int* ul = w.ulist + size_t(t) * m;
  const size_t row0 = size_t(t) * p.n_tok + p.off;  // feature row of patch 0 of this tile
  const float* fin = p.feat[p.fin];
  if (threadIdx.x < SPD_MAX_CLUSTERS) ncl[threadIdx.x] = 0;
  for (int jj = threadIdx.x; jj < nl; jj += blockDim.x) {
    idx[jj] = ul[j0 + jj];
    av[jj] = ordered_val(w.asim[size_t(t) * p.n + ul[j0 + jj]]);
  }
  if (RES && threadIdx.x == 0) {
    mbar_init(&rows_bar, 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (RES && threadIdx.x == 0 && nl > 0) {
    mbar_arrive_expect_tx(&rows_bar, uint32_t(nl) * D * 4);
    for (int jj = 0; jj < nl; ++jj)
      bulk_load(rows + size_t(jj) * D, fin + (row0 + idx[jj]) * D, uint32_t(D) * 4, &rows_bar);
  }
  if (m > 0) {
#pragma unroll 4
    for (int e = threadIdx.x; e < K * D; e += blockDim.x) {
      const int k = e / D, c = e % D;
      cent[e] = feat_row(p, p.fin, t, ul[(k * m) / K])[c];
    }
  }
  if (RES && nl > 0) {
    volatile int no_abort = 0;
    if (!mbar_wait(&rows_bar, 0, &no_abort, kWaitBudget)) {
      set_status(w.status, SPD_ETIMEOUT);
      mbar_wait(&rows_bar, 0, &no_abort, kWaitBudget);  // the copies land before anything reuses it
    }
  }
  __syncthreads();
  // this CTA's token jj of the tile's non-anchor list, row of F^L
  auto xrow = [&](int jj) -> const float* {
    return RES ? rows + size_t(jj) * D : fin + (row0 + idx[jj]) * D;
  };
  for (int it = 0; it < p.iters && m > 0; ++it) {
    // assignment of this CTA's points
    if (threadIdx.x == 0) changed = 0;
    __syncthreads();
    bool done_assign = false;
    // K = 4 with the rows resident: the centroids in registers (242 registers a thread, one CTA an
    // SM). The L2-streaming form takes the loop below instead: at 119 registers two of its CTAs
    // share an SM, which hides more of the row loads' latency (64 tiles: 780 -> 606 us a call).
    if constexpr (KN == 4 && RES) {
      if (D <= 1024) {
        done_assign = true;
        // lane's columns 4 lane + 128 j (j < 8) of the four centroids in registers
        float4 cr[4][8];
#pragma unroll
        for (int k = 0; k < 4; ++k)
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int c = 4 * lane + 128 * j;
            cr[k][j] = (k < K && c < D) ? *reinterpret_cast<const float4*>(cent + k * D + c)
                                        : make_float4(0.f, 0.f, 0.f, 0.f);
          }
        for (int jj = warp; jj < nl; jj += nw) {
          const float* x = xrow(jj);
          float4 xv[8];
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            const int c = 4 * lane + 128 * j;
            xv[j] = c < D ? *reinterpret_cast<const float4*>(x + c) : make_float4(0.f, 0.f, 0.f, 0.f);
          }
          float pd[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
          for (int j = 0; j < 8; ++j)
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float d0 = xv[j].x - cr[k][j].x, d1 = xv[j].y - cr[k][j].y,
                          d2 = xv[j].z - cr[k][j].z, d3 = xv[j].w - cr[k][j].w;
              pd[k] += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
            }
          int best = 0;
          float bd = 0.0f;
#pragma unroll
          for (int k = 0; k < 4; ++k)
            if (k < K) {
              const float dk = warp_sum(pd[k]);
              if (k == 0 || dk < bd) {
                bd = dk;
                best = k;
              }
            }
          if (lane == 0) {
            if (it == 0 || asg[jj] != best) changed = 1;
            asg[jj] = int8_t(best);
          }
        }
      }
    }
    for (int jj = done_assign ? nl : warp; jj < nl; jj += nw) {
      const float* x = xrow(jj);
      float part_d[KN];
#pragma unroll
      for (int k = 0; k < KN; ++k) part_d[k] = 0.0f;
      // 16-byte loads, four in flight per lane (D is a multiple of 4)
      for (int cb = 4 * lane; cb < D; cb += 512) {
        float4 xv[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = cb + 128 * u;
          xv[u] = c < D ? *reinterpret_cast<const float4*>(x + c) : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
          const int c = cb + 128 * u;
          if (c < D) {
#pragma unroll
            for (int k = 0; k < KN; ++k)
              if (k < K) {
                const float4 ce = *reinterpret_cast<const float4*>(cent + k * D + c);
                const float d0 = xv[u].x - ce.x, d1 = xv[u].y - ce.y, d2 = xv[u].z - ce.z,
                            d3 = xv[u].w - ce.w;
                part_d[k] += d0 * d0 + d1 * d1 + d2 * d2 + d3 * d3;
              }
          }
        }
      }
      int best = 0;
      float bd = 0.0f;
#pragma unroll
      for (int k = 0; k < KN; ++k)
        if (k < K) {
          const float dk = warp_sum(part_d[k]);
          if (k == 0 || dk < bd) {
            bd = dk;
            best = k;
          }
        }
      if (lane == 0) {
        if (it == 0 || asg[jj] != best) changed = 1;
        asg[jj] = int8_t(best);
      }
    }
    __syncthreads();
    // this CTA's column sums (token order, in registers) and sizes
    if (threadIdx.x < K) cnt[threadIdx.x] = 0;
    __syncthreads();
    for (int jj = threadIdx.x; jj < nl; jj += blockDim.x) atomicAdd(&cnt[asg[jj]], 1);
    column_sums<KN>(part, K, D, nl, asg,
                    RowAccess{RES ? rows : nullptr, fin, row0, idx, D, nullptr});
    cl.sync();
    // one warp reads the peers' flags and sizes (lane r: CTA r) and publishes them in this CTA
    if (warp == 0) {
      const int f = lane < KC ? *cl.map_shared_rank(&changed, lane) : 0;
      const int any = __any_sync(0xffffffffu, f != 0);
      for (int k = 0; k < K; ++k) {
        int n = lane < KC ? cl.map_shared_rank(cnt, lane)[k] : 0;
#pragma unroll
        for (int off = 16; off; off >>= 1) n += __shfl_xor_sync(0xffffffffu, n, off);
        if (lane == 0) ncl[k] = n;
      }
      if (lane == 0) any_changed = any;
    }
    __syncthreads();
    if (it > 0 && !any_changed) break;  // cluster-uniform decision
    // new centroids for this CTA's column slice, written into every CTA
    cluster_column_reduce<KC>(cl, part, K, D, rank, [&](int k, int c, float sum) {
      const int n = ncl[k];
      const float v = n > 0 ? sum / float(n) : cent[k * D + c];
      for (int rr = 0; rr < KC; ++rr) cl.map_shared_rank(cent, rr)[k * D + c] = v;
    });
    cl.sync();
  }
  // final assignment: sizes, the per-cluster sums of a_j, and the assignment itself
  if (threadIdx.x < K) {
    cnt[threadIdx.x] = 0;
    asum_part[threadIdx.x] = 0.0f;
  }
  __syncthreads();
  for (int jj = threadIdx.x; jj < nl; jj += blockDim.x) {
    atomicAdd(&cnt[asg[jj]], 1);
    w.assign[size_t(t) * m + j0 + jj] = asg[jj];
  }
  if (threadIdx.x == 0)  // token order
    for (int jj = 0; jj < nl; ++jj) asum_part[asg[jj]] += av[jj];
  // per layer: sums over each cluster of unit feature rows (F_l,j / ||F_l,j||), or of raw rows and
  // of st1 for the MSE and KL similarities
  // (RES: the final layer first, from the resident rows; then each other layer's rows are copied
  // into the same buffer)
  constexpr bool cos_sim = COS;
  for (int li = 0; li < p.L; ++li) {
    const int l = RES ? (li == 0 ? p.fin : (li <= p.fin ? li - 1 : li)) : li;
    const float* rstat = (cos_sim ? w.inv : w.st1) + (size_t(l) * p.n_tiles + t) * p.n;
    const float* fl = p.feat[l];
    __syncthreads();  // the previous layer's rows are no longer read
    for (int jj = threadIdx.x; jj < nl; jj += blockDim.x) rinv[jj] = rstat[idx[jj]];
    if (RES && l != p.fin && threadIdx.x == 0 && nl > 0) {
      mbar_arrive_expect_tx(&rows_bar, uint32_t(nl) * D * 4);
      for (int jj = 0; jj < nl; ++jj)
        bulk_load(rows + size_t(jj) * D, fl + (row0 + idx[jj]) * D, uint32_t(D) * 4, &rows_bar);
    }
    if (RES && l != p.fin && nl > 0) {
      volatile int no_abort = 0;
      if (!mbar_wait(&rows_bar, li & 1, &no_abort, kWaitBudget)) {
        set_status(w.status, SPD_ETIMEOUT);
        mbar_wait(&rows_bar, li & 1, &no_abort, kWaitBudget);
      }
    }
    __syncthreads();
    if (!cos_sim && threadIdx.x == 0) {  // token order, fp64 (KL: the fp64 log-sum-exps)
      const float* lo = p.sim == SPD_SIM_KL ? w.st3 + (size_t(l) * p.n_tiles + t) * p.n : nullptr;
      for (int k = 0; k < K; ++k) ssum_part[k] = 0.0;
      for (int jj = 0; jj < nl; ++jj)
        ssum_part[asg[jj]] += double(rinv[jj]) + (lo ? double(lo[idx[jj]]) : 0.0);
    }
    column_sums<KN>(part, K, D, nl, asg,
                    RowAccess{RES ? rows : nullptr, fl, row0, idx, D, cos_sim ? rinv : static_cast<float*>(nullptr)});
    cl.sync();
    float* csum = w.csum + (size_t(t) * p.L + l) * K * D;
    cluster_column_reduce<KC>(cl, part, K, D, rank, [&](int k, int c, float sum) {
      csum[k * D + c] = sum;
      if constexpr (FUSED)  // the layer's cluster sums into every CTA (the centroids are done)
        for (int rr = 0; rr < KC; ++rr) cl.map_shared_rank(cent, rr)[k * D + c] = sum;
    });
    if (!cos_sim && rank == 0 && warp == 1) {  // CTA sums added in rank order
      for (int k = 0; k < K; ++k) {
        const double sr = lane < KC ? cl.map_shared_rank(ssum_part, lane)[k] : 0.0;
        double a = 0.0;
        for (int rr = 0; rr < KC; ++rr) a += __shfl_sync(0xffffffffu, sr, rr);
        if (lane == 0) w.ssum[(size_t(t) * p.L + l) * 16 + k] = a;
      }
    }
    if (FUSED && li == p.L - 1 && warp == 2) {
      // every CTA: the cluster's sums of a_j over the CTAs, in rank order (lane r reads CTA r)
      float ar[SPD_MAX_CLUSTERS];  // all of CTA lane's sums first (one remote round trip)
      const float* peer = lane < KC ? cl.map_shared_rank(asum_part, lane) : nullptr;
      for (int k = 0; k < K; ++k) ar[k] = peer ? peer[k] : 0.0f;
      for (int k = 0; k < K; ++k) {
        float a = 0.0f;
        for (int rr = 0; rr < KC; ++rr) a += __shfl_sync(0xffffffffu, ar[k], rr);
        if (lane == 0) ak[k] = a;
      }
    }
    if (li == p.L - 1 && rank == 0 && warp == 0) {
      // sizes and a_j sums over the CTAs (lane r reads CTA r; the a_j sums added in rank order)
      int sizes[SPD_MAX_CLUSTERS], q[SPD_MAX_CLUSTERS];
      for (int k = 0; k < K; ++k) {
        const int nr = lane < KC ? cl.map_shared_rank(cnt, lane)[k] : 0;
        const float ar = lane < KC ? cl.map_shared_rank(asum_part, lane)[k] : 0.0f;
        int n = nr;
#pragma unroll
        for (int off = 16; off; off >>= 1) n += __shfl_xor_sync(0xffffffffu, n, off);
        float a = 0.0f;
        for (int rr = 0; rr < KC; ++rr) a += __shfl_sync(0xffffffffu, ar, rr);
        sizes[k] = n;
        if (lane == 0) {
          w.counts[t * 16 + k] = n;
          w.asum[t * 16 + k] = a;
        }
      }
      if (lane == 0) {
        compute_quotas(sizes, K, p.n_cmp, q);
        for (int k = 0; k < K; ++k) w.quotas[t * 16 + k] = q[k];
      }
    }
    cl.sync();  // peers' shared memory is read above; keep it alive and unchanged until here
    if constexpr (FUSED) {
      // this CTA's tokens: f_i.(S_l,k - f_i) with f = F / |F| from the resident rows of layer l
      const float wl = (l == p.fin) ? p.wf : p.w[l];
      for (int jj = warp; jj < nl; jj += nw) {
        if (li == 0 && lane == 0) sacc[jj] = 0.0f;
        if (wl == 0.0f) continue;
        const float* x = rows + size_t(jj) * D;
        const float* sk = cent + size_t(asg[jj]) * D;
        const float iv = rinv[jj];
        float dot = 0.0f;
        for (int c = 4 * lane; c < D; c += 128) {
          const float4 xv = *reinterpret_cast<const float4*>(x + c);
          const float4 sv = *reinterpret_cast<const float4*>(sk + c);
          const float b0 = xv.x * iv, b1 = xv.y * iv, b2 = xv.z * iv, b3 = xv.w * iv;
          dot += b0 * (sv.x - b0) + b1 * (sv.y - b1) + b2 * (sv.z - b2) + b3 * (sv.w - b3);
        }
        dot = warp_sum(dot);
        if (lane == 0) sacc[jj] += wl * dot;
      }
    }
  }
  if constexpr (FUSED) fused_select<KC>(p, w, out, cl, rank, t, j0, nl, asg, idx, av, sacc, ncl, ak,
                                        reinterpret_cast<uint64_t*>(rows));
}

// ---- 6. per-token Eq. 3 scores ----------------------------------------------------------------
// Per layer, with X_k the cluster's column sums and c = |C_k|, the sum over the other members j:
//   cos: sum_j f_i.f_j = f_i.(X_k - f_i)                                     (f = F / |F|)
//   MSE: sum_j -|F_i - F_j|^2 / d = -[(c - 1) |F_i|^2 - 2 F_i.(X_k - F_i) + (Q_k - |F_i|^2)] / d
//   KL:  sum_j -KL(P_i || P_j) = -c sum_c P_i,c (log P_i,c - (X_k,c - S_k) / c)
//        (the j = i term is 0; (X_k - S_k) / c is the cluster mean of log P_j, so every product
//        is of a probability and an O(1) difference of logs, with no cancellation of large sums)
// (Q_k, S_k: the cluster's sums of |F_j|^2 and of lse_j.)
// One warp per token. The cosine instance is held to 80 registers so that three CTAs share an SM
// (a few bytes of spills; 64 tiles about 10 us faster than at 97 registers and two CTAs).
template <int SIM>
__global__ void __launch_bounds__(256, SIM == SPD_SIM_COS ? 3 : 1) score_kernel(PruneDims p, PruneWs w) {
  pdl_launch_dependents();
  pdl_wait();
  const int t = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int j = blockIdx.x * 8 + warp;
  if (j >= p.m) return;
  const int i = w.ulist[size_t(t) * p.m + j];
  const int k = w.assign[size_t(t) * p.m + j];
  const int cnt = w.counts[t * 16 + k];
  const float ai = ordered_val(w.asim[size_t(t) * p.n + i]);
  float s;
  if (cnt <= 1) {
    s = p.wa * 2.0f * ai;
  } else {
    float acc = 0.0f;
    for (int l = 0; l < p.L; ++l) {
      const float wl = (l == p.fin) ? p.wf : p.w[l];
      if (wl == 0.0f) continue;
      const float4* x4 = reinterpret_cast<const float4*>(feat_row(p, l, t, i));
      const size_t so = (size_t(l) * p.n_tiles + t) * p.n + i;
      const float iv = SIM == SPD_SIM_COS ? w.inv[so] : 1.0f;
      // KL in fp64: log P_i,c = x_c - lse_i and the cluster mean of log P_j,c
      const double lse = SIM == SPD_SIM_KL ? double(w.st1[so]) + double(w.st3[so]) : 0.0;
      const double sbar = SIM == SPD_SIM_KL ? w.ssum[(size_t(t) * p.L + l) * 16 + k] / double(cnt) : 0.0;
      const float4* c4 =
          reinterpret_cast<const float4*>(w.csum + ((size_t(t) * p.L + l) * p.K + k) * p.d);
      // 16-byte loads, sixteen in flight per lane, two independent chains
      const int d4 = p.d / 4;
      float dot0 = 0.0f, dot1 = 0.0f;
      double kdot = 0.0;  // KL
      for (int cb = lane; cb < d4; cb += 256) {
        float4 xv[8], cv[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          const int c = cb + 32 * u;
          xv[u] = c < d4 ? x4[c] : make_float4(0.f, 0.f, 0.f, 0.f);
          cv[u] = c < d4 ? c4[c] : make_float4(0.f, 0.f, 0.f, 0.f);
        }
#pragma unroll
        for (int u = 0; u < 8; ++u) {
          // cos: f.(X - f) with f = x |x|^-1; MSE: x.(X - x); KL: P.(log P - mean_j log P_j)
          const float b0 = xv[u].x * iv, b1 = xv[u].y * iv, b2 = xv[u].z * iv, b3 = xv[u].w * iv;
          if constexpr (SIM == SPD_SIM_KL) {
            if (cb + 32 * u >= d4) continue;  // a zero-filled slot is no zero term here
            const double dn = double(cnt);
            const double l0 = double(b0) - lse, l1 = double(b1) - lse, l2 = double(b2) - lse,
                         l3 = double(b3) - lse;
            kdot += exp(l0) * (l0 - (double(cv[u].x) / dn - sbar)) +
                    exp(l1) * (l1 - (double(cv[u].y) / dn - sbar)) +
                    exp(l2) * (l2 - (double(cv[u].z) / dn - sbar)) +
                    exp(l3) * (l3 - (double(cv[u].w) / dn - sbar));
          } else {
            const float part =
                b0 * (cv[u].x - b0) + b1 * (cv[u].y - b1) + b2 * (cv[u].z - b2) + b3 * (cv[u].w - b3);
            if (u & 1) dot1 += part;
            else dot0 += part;
          }
        }
      }
      const float dot = warp_sum(dot0 + dot1);
      float term = dot;
      if (SIM == SPD_SIM_MSE) {
        const float sk = float(w.ssum[(size_t(t) * p.L + l) * 16 + k]), st = w.st1[so];
        term = -(float(cnt - 1) * st - 2.0f * dot + (sk - st)) / float(p.d);
      } else if (SIM == SPD_SIM_KL) {
        term = float(-double(cnt) * warp_sum_d(kdot));
      }
      acc += wl * term;
    }
    const float inv_c = 1.0f / float(cnt - 1);
    s = acc * inv_c + p.wa * (ai + (w.asum[t * 16 + k] - ai) * inv_c);
  }
  if (lane == 0) w.score[size_t(t) * p.m + j] = s;
}

// ---- received attention from full maps (Sec. 4.1.1 without [CLS]) ------------------------------
// Column sums of attention maps: CTA (column block, map, row split) adds rows [q0, q1) of its 1024
// columns (thread: four adjacent columns, float4 loads, eight rows in flight) in row order.
__global__ void __launch_bounds__(256) received_colsum_kernel(const float* maps, int n_q,
                                                              int n_k, int rows_per_split,
                                                              float* __restrict__ partial) {
  pdl_launch_dependents();
  pdl_wait();
  const int c4 = blockIdx.x * 256 + threadIdx.x;  // float4 column group
  const int mp = blockIdx.y, sp = blockIdx.z, n_maps = gridDim.y;
  if (4 * c4 >= n_k) return;
  const int q0 = sp * rows_per_split, q1 = min(n_q, q0 + rows_per_split);
  const float4* src = reinterpret_cast<const float4*>(maps + size_t(mp) * n_q * n_k) + c4;
  const size_t ld4 = n_k / 4;
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int q = q0; q < q1; q += 8) {
    float4 v[8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
      v[u] = q + u < q1 ? __ldcs(src + size_t(q + u) * ld4) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
      acc.x += v[u].x;
      acc.y += v[u].y;
      acc.z += v[u].z;
      acc.w += v[u].w;
    }
  }
  reinterpret_cast<float4*>(partial + (size_t(sp) * n_maps + mp) * n_k)[c4] = acc;
}

// out[m][j] = sum over the members i of group j (ascending) of (sum over splits, in order, of the
// partial column sums) / n_q; without groups j = i.
__global__ void __launch_bounds__(256) received_finish_kernel(const float* partial,
                                                              int n_maps, int n_k, int n_splits,
                                                              float inv_nq,
                                                              const int32_t* gstart,
                                                              const int32_t* gmem,
                                                              int n_out, float* __restrict__ out,
                                                              int* status) {
  pdl_launch_dependents();
  pdl_wait();
  const int j = blockIdx.x * 256 + threadIdx.x, mp = blockIdx.y;
  if (j >= n_out) return;
  auto col = [&](int i) {
    float s = 0.0f;
    for (int sp = 0; sp < n_splits; ++sp) s += partial[(size_t(sp) * n_maps + mp) * n_k + i];
    return s * inv_nq;
  };
  float v = 0.0f;
  if (gstart) {
    for (int e = gstart[j]; e < gstart[j + 1]; ++e) {
      const int i = gmem[e];
      if (i < 0 || i >= n_k) {
        set_status(status, SPD_EINVAL);
        continue;
      }
      v += col(i);
    }
  } else {
    v = col(j);
  }
  out[size_t(mp) * n_out + j] = v;
}

// ---- 7. per-cluster bottom-N_k, compaction, outputs -------------------------------------------
__global__ void __launch_bounds__(1024) select_kernel(PruneDims p, PruneWs w, int32_t* keep_idx,
                                                      uint8_t* kind, int8_t* cluster, float* scores) {
  pdl_launch_dependents();
  pdl_wait();
  __shared__ uint64_t keys[4096];
  __shared__ uint8_t kept[4096];
  __shared__ int tmp[32];
  __shared__ int seg[SPD_MAX_CLUSTERS + 1];
  __shared__ int quota[SPD_MAX_CLUSTERS];
  const int t = blockIdx.x, m = p.m;
  const int* ul = w.ulist + size_t(t) * m;
  int N = 1;
  while (N < max(m, 1)) N <<= 1;
  for (int j = threadIdx.x; j < N; j += blockDim.x) {
    uint64_t key = ~0ull;
    if (j < m)
      key = (uint64_t(w.assign[size_t(t) * m + j]) << 45) |
            (uint64_t(ordered_key(w.score[size_t(t) * m + j])) << 13) | uint64_t(ul[j]);
    keys[j] = key;
  }
  for (int i = threadIdx.x; i < p.n; i += blockDim.x) kept[i] = uint8_t(w.role[size_t(t) * p.n + i]);
  if (threadIdx.x == 0) {
    int acc = 0;
    for (int k = 0; k < p.K; ++k) {
      seg[k] = acc;
      acc += w.counts[t * 16 + k];
      quota[k] = w.quotas[t * 16 + k];
    }
    seg[p.K] = acc;
  }
  __syncthreads();
  if (m <= kRankMax) {
    // the key at sorted position r of cluster k's segment is kept iff r - seg[k] < quota[k]
    rank_keys(keys, m, [&](int j, int r) {
      const int k = int(keys[j] >> 45);
      if (r - seg[k] < quota[k]) kept[keys[j] & 0x1fffu] = 2;
    });
  } else {
    bitonic_sort(keys, N);
    for (int r = threadIdx.x; r < m; r += blockDim.x) {
      const int k = int(keys[r] >> 45);
      if (r - seg[k] < quota[k]) kept[keys[r] & 0x1fffu] = 2;
    }
  }
  __syncthreads();
  const int base = threadIdx.x * 4;
  int nk = 0;
  for (int q = 0; q < 4; ++q)
    if (base + q < p.n) nk += kept[base + q] != 0;
  int pos = block_scan_excl(nk, tmp, nullptr);
  for (int q = 0; q < 4; ++q) {
    const int i = base + q;
    if (i >= p.n) break;
    if (kept[i]) {
      if (pos < p.keep) keep_idx[size_t(t) * p.keep + pos] = i;
      else set_status(w.status, SPD_EINVAL);
      ++pos;
    }
    if (kind) kind[size_t(t) * p.n + i] = kept[i];
    if (kept[i] == 1) {
      if (cluster) cluster[size_t(t) * p.n + i] = -1;
      if (scores) scores[size_t(t) * p.n + i] = INFINITY;
    }
  }
  for (int j = threadIdx.x; j < m; j += blockDim.x) {
    if (cluster) cluster[size_t(t) * p.n + ul[j]] = int8_t(w.assign[size_t(t) * m + j]);
    if (scores) scores[size_t(t) * p.n + ul[j]] = w.score[size_t(t) * m + j];
  }
}

__global__ void gather_bf16_kernel(const float* src, int n_tok, int d, int off, const int32_t* idx,
                                   int keep,
                                   __nv_bfloat16* __restrict__ dst, int* status) {
  pdl_launch_dependents();
  pdl_wait();
  const int j = blockIdx.x, t = blockIdx.y;
  const int i = idx[size_t(t) * keep + j];
  if (i < 0 || i >= n_tok - off) {
    if (threadIdx.x == 0) set_status(status, SPD_EINVAL);
    return;
  }
  const float4* s = reinterpret_cast<const float4*>(src + (size_t(t) * n_tok + off + i) * d);
  uint2* o = reinterpret_cast<uint2*>(dst + (size_t(t) * keep + j) * d);
  for (int c = threadIdx.x; c < d / 4; c += blockDim.x) {
    const float4 v = s[c];
    __nv_bfloat162 lo = __floats2bfloat162_rn(v.x, v.y), hi = __floats2bfloat162_rn(v.z, v.w);
    o[c] = make_uint2(*reinterpret_cast<uint32_t*>(&lo), *reinterpret_cast<uint32_t*>(&hi));
  }
}

int validate(const spd_prune_cfg* c, PruneDims* p) {
  if (!c) return fail(SPD_EINVAL, "null prune config");
  if (c->n_tiles < 1 || c->n_layers < 1 || c->n_layers > SPD_MAX_FEAT_LAYERS)
    return fail(SPD_EINVAL, "n_tiles >= 1 and n_layers in [1, %d] required", SPD_MAX_FEAT_LAYERS);
  if (c->final_layer < 0 || c->final_layer >= c->n_layers) return fail(SPD_EINVAL, "bad final_layer");
  const int off = c->has_cls ? 1 : 0;
  const int n = c->n_tok - off;
  if (n < 1 || n > 4096) return fail(SPD_EINVAL, "patch count must lie in [1, 4096]");
  if (c->d_feat < 4 || c->d_feat % 4 || c->d_feat > 4096)
    return fail(SPD_EINVAL, "d_feat must be a multiple of 4 in [4, 4096]");
  if (c->n_heads < 1) return fail(SPD_EINVAL, "n_heads >= 1 required");
  if (c->attn_form != 0 && c->attn_form != 1) return fail(SPD_EINVAL, "attn_form must be 0 or 1");
  if (c->attn_form == 0 && !c->has_cls) return fail(SPD_EINVAL, "CLS-row attention needs has_cls");
  if (c->keep < 1 || c->keep > n) return fail(SPD_EINVAL, "keep must lie in [1, n_patch]");
  if (c->n_clusters < 1 || c->n_clusters > SPD_MAX_CLUSTERS) return fail(SPD_EINVAL, "bad n_clusters");
  if (size_t(c->n_clusters) * c->d_feat > 24576)
    return fail(SPD_EINVAL, "n_clusters * d_feat must not exceed 24576");
  if (c->kmeans_iters < 1) return fail(SPD_EINVAL, "kmeans_iters >= 1 required");
  if (!(c->anchor_ratio >= 0.0 && c->anchor_ratio <= 1.0))
    return fail(SPD_EINVAL, "anchor_ratio must lie in [0, 1]");
  if (c->sim_kind < SPD_SIM_COS || c->sim_kind > SPD_SIM_KL) return fail(SPD_EINVAL, "bad sim_kind");
  if (c->ablate & ~(SPD_PRUNE_NO_FINAL_SIM | SPD_PRUNE_NO_ANCHOR_SIM))
    return fail(SPD_EINVAL, "unknown ablate bits");
  p->sim = c->sim_kind;
  p->wf = (c->ablate & SPD_PRUNE_NO_FINAL_SIM) ? 0.0f : 1.0f;
  p->wa = (c->ablate & SPD_PRUNE_NO_ANCHOR_SIM) ? 0.0f : 1.0f;
  p->n_tiles = c->n_tiles;
  p->n_tok = c->n_tok;
  p->off = off;
  p->n = n;
  p->d = c->d_feat;
  p->L = c->n_layers;
  p->fin = c->final_layer;
  p->H = c->n_heads;
  p->form = c->attn_form;
  p->n_att = c->attn_form == 0 ? c->n_tok : n;
  p->keep = c->keep;
  p->K = c->n_clusters;
  p->iters = c->kmeans_iters;
  p->n_anc = int(floor(double(c->keep) * c->anchor_ratio + 0.5));
  if (p->n_anc > c->keep) p->n_anc = c->keep;
  p->n_cmp = c->keep - p->n_anc;
  p->m = n - p->n_anc;
  for (int l = 0; l < SPD_MAX_FEAT_LAYERS; ++l) {
    p->w[l] = c->layer_weight[l];
    p->feat[l] = nullptr;
  }
  return SPD_OK;
}

PruneWs carve(const PruneDims& p, Carve& cv) {
  PruneWs w;
  const size_t T = p.n_tiles;
  w.status = cv.status();
  w.a_v = cv.take<float>(T * p.n);
  w.inv = cv.take<float>(T * p.n * p.L);
  const size_t nst = p.sim == SPD_SIM_COS ? 0 : T * p.n * p.L;
  w.st1 = cv.take<float>(nst);
  w.st2 = cv.take<float>(p.sim == SPD_SIM_KL ? nst : 0);
  w.st3 = cv.take<float>(p.sim == SPD_SIM_KL ? nst : 0);
  w.role = cv.take<int8_t>(T * p.n);
  w.alist = cv.take<int32_t>(T * (p.n_anc + 1));
  w.ulist = cv.take<int32_t>(T * (p.m + 1));
  w.asim = cv.take<uint32_t>(T * p.n);
  w.assign = cv.take<int32_t>(T * (p.m + 1));
  w.counts = cv.take<int32_t>(T * 16);
  w.quotas = cv.take<int32_t>(T * 16);
  w.asum = cv.take<float>(T * 16);
  w.csum = cv.take<float>(T * p.L * p.K * p.d);
  w.ssum = cv.take<double>(T * p.L * 16);
  w.score = cv.take<float>(T * (p.m + 1));
  return w;
}

constexpr size_t kResSmem = 200 * 1024;  // dynamic shared memory of the resident K-means
int g_res_clusters = -1;                 // 16-CTA clusters of it the GPU holds at once

template <int KC, bool RES, int KN, bool FUSED = false>
cudaError_t launch_kmeans(const PruneDims& p, const PruneWs& w, const PruneOut& out, size_t smem,
                          cudaStream_t st) {
  auto kern = FUSED ? kmeans_kernel<KC, RES, KN, true, FUSED>
              : p.sim == SPD_SIM_COS ? kmeans_kernel<KC, RES, KN, true> : kmeans_kernel<KC, RES, KN, false>;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(KC, p.n_tiles);
  cfg.blockDim = dim3(kmeans_threads<KN>());
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = KC;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, kern, p, w, out);
}

// Kernel attributes (once per process) and whether 16-CTA clusters of the resident kernel fit.
int kmeans_setup() {
  static std::once_flag once;
  static cudaError_t err = cudaSuccess;
  std::call_once(once, [] {
    auto streamed = [](auto kern) {
      return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, 2 * 24576 * 4);
    };
    auto resident = [](auto kern) {
      cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kResSmem));
      return e;
    };
    err = streamed(kmeans_kernel<8, false, 4, true>);
    if (err == cudaSuccess) err = streamed(kmeans_kernel<4, false, 4, true>);
    if (err == cudaSuccess) err = streamed(kmeans_kernel<4, false, 4, false>);
    if (err == cudaSuccess) err = streamed(kmeans_kernel<8, false, SPD_MAX_CLUSTERS, true>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, 4, true>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, SPD_MAX_CLUSTERS, true>);
    if (err == cudaSuccess) err = streamed(kmeans_kernel<8, false, 4, false>);
    if (err == cudaSuccess) err = streamed(kmeans_kernel<8, false, SPD_MAX_CLUSTERS, false>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, 4, false>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, SPD_MAX_CLUSTERS, false>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, 4, true, true>);
    if (err == cudaSuccess) err = resident(kmeans_kernel<16, true, SPD_MAX_CLUSTERS, true, true>);
    g_res_clusters = 0;
    if (err == cudaSuccess) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(16);
      cfg.blockDim = dim3(512);
      cfg.dynamicSmemBytes = kResSmem;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = 16;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n, kmeans_kernel<16, true, SPD_MAX_CLUSTERS, true>, &cfg) !=
          cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      g_res_clusters = n;
    }
  });
  if (err != cudaSuccess) return fail(SPD_ECUDA, "K-means attributes: %s", cudaGetErrorString(err));
  return SPD_OK;
}

// Which kernels spd_prune launches for p (after kmeans_setup).
struct PrunePlan {
  bool anchor_sim, res, fused;
  int launches;
};
PrunePlan prune_plan(const PruneDims& p) {
  PrunePlan q;
  q.anchor_sim = p.n_anc > 0 && p.m > 0 && p.wa != 0.0f;
  const size_t cent_bytes = size_t(2) * p.K * p.d * sizeof(float);
  const size_t res_bytes = size_t((p.m + 15) / 16) * p.d * sizeof(float) + cent_bytes;
  // K-means: the rows resident in shared memory over 16 CTAs per tile where they fit and all tiles
  // run in one wave of such clusters (latency); else re-read from L2 each pass by 8 CTAs per tile,
  // twice as many tiles at once (throughput), or by 4 where 8-CTA clusters would take more than one
  // wave at two CTAs an SM (the paper's K = 4)
  q.res = p.m > 0 && res_bytes <= kResSmem && g_res_clusters > 0 && p.n_tiles <= g_res_clusters;
  // resident rows and the cosine kind: scores, selection and compaction in the same kernel (CTA 0's
  // row buffer holds the m sort keys and the n kept flags by then)
  const size_t row_bytes = size_t((p.m + 15) / 16) * p.d * sizeof(float);
  q.fused = q.res && p.sim == SPD_SIM_COS && (p.m + 15) / 16 <= 512 &&
            row_bytes >= size_t(8) * (p.m + 1) + p.n;
  q.launches = 2 + int(q.anchor_sim) + 1 + (q.fused ? 0 : int(p.m > 0) + 1);
  return q;
}

}  // namespace
}  // namespace spd

using namespace spd;

extern "C" int spd_prune_launches(const spd_prune_cfg* cfg) {
  PruneDims p;
  if (int rc = validate(cfg, &p)) return rc;
  if (int rc = kmeans_setup()) return rc;
  return prune_plan(p).launches;
}

extern "C" size_t spd_prune_workspace_size(const spd_prune_cfg* cfg) {
  PruneDims p;
  if (validate(cfg, &p)) return 0;
  Carve cv(nullptr, ~size_t(0));
  carve(p, cv);
  return cv.used;
}

extern "C" int spd_prune(const spd_prune_cfg* cfg, const float* const* feats, const float* attn,
                         int32_t* keep_idx, uint8_t* kind, int8_t* cluster, float* scores, void* ws,
                         size_t ws_bytes, void* stream_) {
  PruneDims p;
  if (int rc = validate(cfg, &p)) return rc;
  if (!feats || !attn || !keep_idx || !ws) return fail(SPD_EINVAL, "null buffer");
  for (int l = 0; l < p.L; ++l) {
    if (!feats[l] || (reinterpret_cast<uintptr_t>(feats[l]) & 15))
      return fail(SPD_EINVAL, "feature pointer %d null or not 16-byte aligned", l);
    p.feat[l] = feats[l];
  }
  Carve cv(ws, ws_bytes);
  PruneWs w = carve(p, cv);
  if (!cv.fits()) return fail(SPD_ENOSPC, "prune workspace too small (%zu < %zu)", ws_bytes, cv.used);
  cudaStream_t st = static_cast<cudaStream_t>(stream_);
  const int T = p.n_tiles;
  const int slot = trace_begin(st);
  SPD_CUDA_TRY(launch_pdl(p.sim == SPD_SIM_COS ? rowstats_kernel<SPD_SIM_COS>
                          : p.sim == SPD_SIM_MSE ? rowstats_kernel<SPD_SIM_MSE> : rowstats_kernel<SPD_SIM_KL>,
                          dim3((p.n + 7) / 8, T), dim3(256), 0, st, p, attn, w));
  SPD_CUDA_TRY(launch_pdl(anchor_kernel, dim3(T), dim3(1024), 0, st, p, w));
  if (int rc = kmeans_setup()) return rc;
  const PrunePlan plan = prune_plan(p);
  if (plan.anchor_sim) {
    // the feature dimension over 8 CTAs while the tiles leave most SMs idle, else over 4
    const dim3 g((p.m + 63) / 64, (p.n_anc + 63) / 64, T);
    if (size_t(g.x) * g.y * T * 8 <= 2 * size_t(num_sms()))
      SPD_CUDA_TRY(launch_pdl(p.sim == SPD_SIM_COS ? anchor_sim_kernel<SPD_SIM_COS, 8>
                              : p.sim == SPD_SIM_MSE ? anchor_sim_kernel<SPD_SIM_MSE, 8>
                                                     : anchor_sim_kernel<SPD_SIM_KL, 8>,
                              dim3(g.x * 8, g.y, T), dim3(256), 0, st, p, w));
    else
      SPD_CUDA_TRY(launch_pdl(p.sim == SPD_SIM_COS ? anchor_sim_kernel<SPD_SIM_COS, 4>
                              : p.sim == SPD_SIM_MSE ? anchor_sim_kernel<SPD_SIM_MSE, 4>
                                                     : anchor_sim_kernel<SPD_SIM_KL, 4>,
                              dim3(g.x * 4, g.y, T), dim3(256), 0, st, p, w));
  }
  const size_t cent_bytes = size_t(2) * p.K * p.d * sizeof(float);
  const size_t res_bytes = size_t((p.m + 15) / 16) * p.d * sizeof(float) + cent_bytes;
  const PruneOut out{keep_idx, kind, cluster, scores};
  if (plan.fused && p.K == 4)
    SPD_CUDA_TRY((launch_kmeans<16, true, 4, true>(p, w, out, res_bytes, st)));
  else if (plan.fused)
    SPD_CUDA_TRY((launch_kmeans<16, true, SPD_MAX_CLUSTERS, true>(p, w, out, res_bytes, st)));
  else if (plan.res && p.K == 4)
    SPD_CUDA_TRY((launch_kmeans<16, true, 4>(p, w, out, res_bytes, st)));
  else if (plan.res)
    SPD_CUDA_TRY((launch_kmeans<16, true, SPD_MAX_CLUSTERS>(p, w, out, res_bytes, st)));
  else if (p.K == 4 && size_t(p.n_tiles) * 8 > 2 * size_t(num_sms()))
    SPD_CUDA_TRY((launch_kmeans<4, false, 4>(p, w, out, cent_bytes, st)));
  else if (p.K == 4)
    SPD_CUDA_TRY((launch_kmeans<8, false, 4>(p, w, out, cent_bytes, st)));
  else
    SPD_CUDA_TRY((launch_kmeans<8, false, SPD_MAX_CLUSTERS>(p, w, out, cent_bytes, st)));
  if (!plan.fused) {
    if (p.m > 0) {
      auto score = p.sim == SPD_SIM_COS ? score_kernel<SPD_SIM_COS>
                   : p.sim == SPD_SIM_MSE ? score_kernel<SPD_SIM_MSE> : score_kernel<SPD_SIM_KL>;
      SPD_CUDA_TRY(launch_pdl(score, dim3((p.m + 7) / 8, T), dim3(256), 0, st, p, w));
    }
    SPD_CUDA_TRY(launch_pdl(select_kernel, dim3(T), dim3(1024), 0, st, p, w, keep_idx, kind, cluster,
                            scores));
  }
  // algorithmic work per tile: every tapped layer's features and the attention read once, the
  // kept indices written; anchor similarities (n - N_anc) N_anc d multiply-adds
  trace_end(slot, st, TR_PRUNE, 2.0 * T * double(p.m) * p.n_anc * p.d,
            T * (4.0 * p.L * double(p.n_tok) * p.d + 4.0 * p.H * p.n_att + 4.0 * p.keep + 6.0 * p.n));
  return SPD_OK;
}

namespace {
int received_splits(int n_maps, int n_q, int n_k) {
  const int blocks = (n_k / 4 + 255) / 256;
  int sp = (2 * num_sms() + blocks * n_maps - 1) / (blocks * n_maps);  // about two CTAs per SM
  sp = std::max(1, std::min(sp, (n_q + 63) / 64));                    // at least 64 rows each
  return sp;
}
}  // namespace

extern "C" size_t spd_received_attention_workspace_size(int n_maps, int n_q, int n_k) {
  if (n_maps < 1 || n_q < 1 || n_k < 4) return 0;
  Carve cv(nullptr, ~size_t(0));
  cv.take<float>(size_t(received_splits(n_maps, n_q, n_k)) * n_maps * n_k);
  return cv.used;
}

extern "C" int spd_received_attention(const float* maps, int n_maps, int n_q, int n_k,
                                      const int32_t* group_start, const int32_t* group_members,
                                      int n_out, float* out, void* ws, size_t ws_bytes,
                                      void* stream_) {
  if (!maps || !out || !ws || n_maps < 1 || n_q < 1 || n_k < 4 || n_k % 4 ||
      (reinterpret_cast<uintptr_t>(maps) & 15))
    return fail(SPD_EINVAL, "bad received-attention arguments (n_k a multiple of 4, maps 16-byte aligned)");
  if ((group_start == nullptr) != (group_members == nullptr))
    return fail(SPD_EINVAL, "group_start and group_members go together");
  if (!group_start && n_out != n_k) return fail(SPD_EINVAL, "without groups n_out must equal n_k");
  if (n_out < 1) return fail(SPD_EINVAL, "n_out >= 1 required");
  const int sp = received_splits(n_maps, n_q, n_k);
  Carve cv(ws, ws_bytes);
  float* partial = cv.take<float>(size_t(sp) * n_maps * n_k);
  if (!cv.fits()) return fail(SPD_ENOSPC, "received-attention workspace too small");
  cudaStream_t st = static_cast<cudaStream_t>(stream_);
  const int rows = (n_q + sp - 1) / sp;
  const int slot = trace_begin(st);
  SPD_CUDA_TRY(launch_pdl(received_colsum_kernel, dim3((n_k / 4 + 255) / 256, n_maps, sp), dim3(256),
                          0, st, maps, n_q, n_k, rows, partial));
  SPD_CUDA_TRY(launch_pdl(received_finish_kernel, dim3((n_out + 255) / 256, n_maps), dim3(256), 0, st,
                          static_cast<const float*>(partial), n_maps, n_k, sp, float(1.0 / n_q),
                          group_start, group_members, n_out, out, cv.status()));
  // algorithmic work: every map entry read once, the result written once
  trace_end(slot, st, TR_PRUNE, double(n_maps) * n_q * n_k,
            4.0 * double(n_maps) * n_q * n_k + 4.0 * double(n_maps) * n_out);
  return SPD_OK;
}

extern "C" int spd_gather_rows_bf16(const float* src, int n_tiles, int n_tok, int d, int row_offset,
                                    const int32_t* idx, int keep, uint16_t* dst, void* ws,
                                    void* stream_) {
  if (!src || !idx || !dst || n_tiles < 1 || keep < 1 || d < 4 || d % 4 || row_offset < 0 ||
      row_offset >= n_tok)
    return fail(SPD_EINVAL, "bad gather arguments");
  SPD_CUDA_TRY(launch_pdl(gather_bf16_kernel, dim3(keep, n_tiles), dim3(128), 0,
                          static_cast<cudaStream_t>(stream_), src, n_tok, d, row_offset, idx, keep,
                          reinterpret_cast<__nv_bfloat16*>(dst), ws ? static_cast<int*>(ws) : nullptr));
  return SPD_OK;
}
