// Variable-length causal attention over packed sequences on the tcgen05 tensor cores, queries
// restricted to the attention-active tokens (VSkip-Attn, Sec. 3.2: a skipped token is not a
// query, but it stays a key and a value for every other token of its sequence).
//
// One CTA = up to 128 active queries of one sequence x one head (the MMA's M = 128 rows):
//   warp 4     TMA producer: the Q tile once, then blocks of 128 keys of K and V into a two-stage
//              ring (128-byte swizzle, boxes of 64 head-dim columns)
//   warp 5     MMA issuer: S = Q K^T into TMEM (kind::f16, fp32), then O += P V with P from shared
//              memory and V read in place as an MN-major operand (the layout its TMA box has)
//   warps 0-3  softmax: thread r owns query row r (TMEM lane r); online softmax in fp32 with exp2;
//              P rounded to bf16 into shared memory as a K-major swizzled operand; O rescaled in
//              TMEM when a row's running maximum grows; at the end O / l goes to HBM in bf16
// S alternates between two TMEM buffers, so S of block j + 1 is computed while the softmax of
// block j reads block j's (two passes: the maximum, then the exponentials, sum and P). A query at
// position p sees keys 0..p of its own sequence. Every wait is bounded (status SPD_ETIMEOUT, no
// hang).
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include <cooperative_groups.h>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace spd {
namespace {

namespace cg = cooperative_groups;

constexpr int kTK = 128;              // keys per block (S columns, K of the PV product)
constexpr uint32_t kBox = 128 * 128;  // one TMA box: 128 rows x 64 bf16
constexpr int kThreads = 192;

template <int HD>
struct AttnSmem {
  static constexpr int kChunks = HD / 64;                       // 64-column boxes per row
  static constexpr uint32_t q = 0;                              // Q tile
  static constexpr uint32_t k = q + kChunks * kBox;             // K stages
  static constexpr uint32_t v = k + 2 * kChunks * kBox;         // V stages
  static constexpr uint32_t p = v + 2 * kChunks * kBox;         // P: two 64-key halves
  static constexpr uint32_t bars = p + 2 * kBox;
  static constexpr uint32_t bytes = bars + 128 + 1024;          // + alignment slack
};

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int HD>
__global__ void __launch_bounds__(kThreads, 1)
    attn_tc_kernel(const __grid_constant__ CUtensorMap map_q,
                   const __grid_constant__ CUtensorMap map_kv, __nv_bfloat16* __restrict__ o,
                   int ldo, const int4* tiles, const int32_t* q_pos, int n_heads, int n_kv_heads,
                   int v_off, float scale_log2, int* status, long long budget,
                   unsigned long long* stamp) {
  using L = AttnSmem<HD>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  uint64_t* q_full = reinterpret_cast<uint64_t*>(smem + L::bars);
  uint64_t* kv_full = q_full + 1;   // [2] K and V block landed
  uint64_t* kv_empty = q_full + 3;  // [2] its PV product has completed
  uint64_t* s_full = q_full + 5;    // [2] S of block j is in TMEM buffer j % 2
  uint64_t* s_free = q_full + 7;    // [2] the softmax warps have read S buffer j % 2
  uint64_t* p_full = q_full + 9;    // P written and O rescaled
  uint64_t* o_done = q_full + 10;   // PV product of the current block completed
  uint64_t* drain = q_full + 11;    // every MMA completed
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_full + 12);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int h = blockIdx.y;
  const int hk = h / (n_heads / n_kv_heads);
  if (threadIdx.x == 0) {
    mbar_init(q_full, 1);
    for (int s = 0; s < 2; ++s) {
      mbar_init(&kv_full[s], 1);
      mbar_init(&kv_empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&s_free[b], 4);  // one arrival per softmax warp
    }
    mbar_init(p_full, 4);
    mbar_init(o_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&map_q);
    prefetch_tmap(&map_kv);
  }
  if (warp == 4) {
    tmem_alloc(tmem_slot, 512);  // S: two buffers, columns [0, 128) and [128, 256); O: [256, 256 + HD)
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  const uint32_t t_o = tmem + 256;  // S buffer b at tmem + 128 b

  // Nothing written by an earlier kernel of the stream is read before the grid dependency wait:
  // under programmatic overlap this kernel's prologue may run while several earlier kernels are
  // still resident, so the tile list and the positions (copied or built by a kernel) are read
  // after it, with coherent loads. Q, K and V come from the previous kernels too.
  pdl_launch_dependents();
  pdl_wait();
  if (threadIdx.x == 0) stamp_start(stamp);
  const int4 tl = tiles[blockIdx.x];
  const int q0 = tl.x, nq = tl.y, kv0 = tl.z, len = tl.w;
  const int p_last = q_pos[q0 + nq - 1];  // positions ascend within a tile
  const int nkb = max(1, min((p_last + kTK) / kTK, (len + kTK - 1) / kTK));
  const int my_pos = threadIdx.x < 128 ? q_pos[q0 + min(int(threadIdx.x), nq - 1)] : 0;

  int issued = 0;  // K/V blocks whose loads the producer issued
  if (warp == 4) {
    if (lane == 0) {
      // ---- TMA producer ----
      const uint64_t pol_q = policy_evict_first(), pol_kv = policy_evict_last();
      mbar_arrive_expect_tx(q_full, L::kChunks * kBox);
      for (int c = 0; c < L::kChunks; ++c)
        tma_load_2d(smem + L::q + c * kBox, &map_q, q_full, h * HD + c * 64, q0, pol_q);
      for (int j = 0; j < nkb; ++j) {
        const int s = j & 1;
        if (j >= 2 && !mbar_wait(&kv_empty[s], ((j >> 1) - 1) & 1, abort_flag, budget)) {
          *abort_flag = 1;
          set_status(status, SPD_ETIMEOUT);
          break;
        }
        mbar_arrive_expect_tx(&kv_full[s], 2 * L::kChunks * kBox);
        for (int c = 0; c < L::kChunks; ++c) {
          const int x = hk * HD + c * 64, y = kv0 + j * kTK;
          tma_load_2d(smem + L::k + (s * L::kChunks + c) * kBox, &map_kv, &kv_full[s], x, y, pol_kv);
          tma_load_2d(smem + L::v + (s * L::kChunks + c) * kBox, &map_kv, &kv_full[s], v_off + x, y,
                      pol_kv);
        }
        issued = j + 1;
      }
    }
  } else if (warp == 5) {
    if (lane == 0) {
      // ---- MMA issuer ----
      const uint32_t id_s = idesc_bf16_f32(128, kTK);
      const uint32_t id_o = idesc_bf16_f32(128, HD) | (1u << 16);  // V is MN-major
      const uint32_t sq = smem_u32(smem + L::q), sp = smem_u32(smem + L::p);
      bool ok = mbar_wait(q_full, 0, abort_flag, budget);
      auto issue_s = [&](int j) -> bool {
        const int s = j & 1;
        if (!mbar_wait(&kv_full[s], (j >> 1) & 1, abort_flag, budget)) return false;
        // S buffer s was last read by the softmax of block j - 2
        if (j > 1 && !mbar_wait(&s_free[s], ((j >> 1) - 1) & 1, abort_flag, budget)) return false;
        tc_fence_after();
        const uint32_t sk = smem_u32(smem + L::k + s * L::kChunks * kBox);
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk) {
          const uint32_t off = (kk >> 2) * kBox + (kk & 3) * 32;
          mma_bf16(tmem + 128 * s, sdesc_k128(sq + off), sdesc_k128(sk + off), id_s, kk > 0 ? 1u : 0u);
        }
        mma_commit(&s_full[s]);
        return true;
      };
      if (ok) ok = issue_s(0);
      for (int j = 0; j < nkb && ok; ++j) {
        if (j + 1 < nkb && !(ok = issue_s(j + 1))) break;
        if (!(ok = mbar_wait(p_full, j & 1, abort_flag, budget))) break;
        tc_fence_after();
        const uint32_t sv = smem_u32(smem + L::v + (j & 1) * L::kChunks * kBox);
#pragma unroll
        for (int kk = 0; kk < kTK / 16; ++kk) {
          const uint64_t ad = sdesc_k128(sp + (kk >> 2) * kBox + (kk & 3) * 32);
          const uint64_t bd = sdesc_mn128(sv + kk * 2048, kBox);
          mma_bf16(t_o, ad, bd, id_o, (j > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(o_done);
        mma_commit(&kv_empty[j & 1]);
      }
      if (!ok) {
        *abort_flag = 1;
        set_status(status, SPD_ETIMEOUT);
      }
      mma_commit(drain);  // arrives once every MMA issued above has completed
      volatile int no_abort = 0;
      if (!mbar_wait(drain, 0, &no_abort, budget)) set_status(status, SPD_ETIMEOUT);
    }
  } else {
    // ---- softmax and epilogue: warp w reads TMEM lanes [32 w, 32 w + 32) ----
    const int r = warp * 32 + lane;  // query row of the tile
    const uint32_t lanes = static_cast<uint32_t>(warp * 32) << 16;
    uint8_t* prow = smem + L::p + r * 128;
    float m_run = -INFINITY, l_run = 0.0f;
    bool ok = true;
    for (int j = 0; j < nkb; ++j) {
      const int sb = j & 1;
      if (!(ok = __all_sync(0xffffffffu, mbar_wait(&s_full[sb], (j >> 1) & 1, abort_flag, budget))))
        break;
      tc_fence_after();
      const uint32_t t_s = tmem + 128 * sb + lanes;
      const int kb = j * kTK;
      // Two passes over the block's S row, 32 columns at a time in rolled loops (small code; the
      // fully unrolled single pass held all 128 values in 254 registers and its first run cost
      // 3 us against 1.4 for the second block): the row maximum, then 2^(s - m), the row sum and
      // P. The next block's S goes to the other TMEM buffer meanwhile.
      float mx = -INFINITY;
#pragma unroll 1
      for (int c = 0; c < kTK / 32; ++c) {
        float v[32];
        tmem_ld32(t_s + c * 32, v);
        float m4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float x = (kb + c * 32 + i <= my_pos) ? v[i] * scale_log2 : -INFINITY;
          m4[i & 3] = fmaxf(m4[i & 3], x);
        }
        mx = fmaxf(mx, fmaxf(fmaxf(m4[0], m4[1]), fmaxf(m4[2], m4[3])));
      }
      const float m_new = fmaxf(m_run, mx);  // finite: block 0 holds key 0 <= every position
      const float corr = exp2f(m_run - m_new);  // 0 on the first block
      if (j > 0) {
        // the previous PV product has completed: P's buffer is free and O can be rescaled
        if (!(ok = __all_sync(0xffffffffu, mbar_wait(o_done, (j - 1) & 1, abort_flag, budget))))
          break;
        tc_fence_after();
        if (__any_sync(0xffffffffu, corr != 1.0f)) {
#pragma unroll 1
          for (int c = 0; c < HD / 32; ++c) {
            float v[32];
            tmem_ld32(t_o + lanes + c * 32, v);
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= corr;
            tmem_st32(t_o + lanes + c * 32, v);
          }
        }
      }
      // P in bf16: row r of a K-major operand in the 128-byte swizzle layout (16-byte unit u of
      // the row at position u ^ (r % 8)), keys [0, 64) and [64, 128) in two boxes
      float rs = 0.0f;
#pragma unroll 1
      for (int c = 0; c < kTK / 32; ++c) {
        float v[32];
        tmem_ld32(t_s + c * 32, v);
        float r4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float x = (kb + c * 32 + i <= my_pos) ? v[i] * scale_log2 : -INFINITY;
          v[i] = exp2f(x - m_new);
          r4[i & 3] += v[i];
        }
        rs += (r4[0] + r4[1]) + (r4[2] + r4[3]);
#pragma unroll
        for (int uu = 0; uu < 4; ++uu) {
          const int u = 4 * c + uu;
          const uint4 w = make_uint4(pack_bf16(v[8 * uu], v[8 * uu + 1]), pack_bf16(v[8 * uu + 2], v[8 * uu + 3]),
                                     pack_bf16(v[8 * uu + 4], v[8 * uu + 5]),
                                     pack_bf16(v[8 * uu + 6], v[8 * uu + 7]));
          *reinterpret_cast<uint4*>(prow + (u >> 3) * kBox + (((u & 7) ^ (r & 7)) << 4)) = w;
        }
      }
      l_run = l_run * corr + rs;
      m_run = m_new;
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s_free[sb]);  // S buffer sb read (both passes)
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(p_full);
    }
    if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_done, (nkb - 1) & 1, abort_flag, budget));
    if (!ok) {
      *abort_flag = 1;
      set_status(status, SPD_ETIMEOUT);
    } else {
      tc_fence_after();
      const float inv = 1.0f / l_run;
      __nv_bfloat16* orow = o + size_t(q0 + r) * ldo + h * HD;
#pragma unroll 1
      for (int c = 0; c < HD / 32; ++c) {
        float v[32];
        tmem_ld32(t_o + lanes + c * 32, v);
        if (r < nq) {
#pragma unroll
          for (int u = 0; u < 4; ++u)
            reinterpret_cast<uint4*>(orow + c * 32)[u] =
                make_uint4(pack_bf16(v[8 * u] * inv, v[8 * u + 1] * inv),
                           pack_bf16(v[8 * u + 2] * inv, v[8 * u + 3] * inv),
                           pack_bf16(v[8 * u + 4] * inv, v[8 * u + 5] * inv),
                           pack_bf16(v[8 * u + 6] * inv, v[8 * u + 7] * inv));
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 128 && *abort_flag) {
    // loads issued but never consumed land before the CTA exits (without an abort the last PV
    // product consumed every issued block)
    volatile int no_abort = 0;
    mbar_wait(q_full, 0, &no_abort, budget);
    for (int j = max(0, issued - 2); j < issued; ++j)
      mbar_wait(&kv_full[j & 1], (j >> 1) & 1, &no_abort, budget);
  }
  __syncwarp();
  tc_fence_after();
  if (warp == 4) tmem_dealloc(tmem, 512);
  if (threadIdx.x == 0) stamp_end(stamp);
}

template <int HD>
int launch(const CUtensorMap& mq, const CUtensorMap& mkv, void* o, int ldo, const int4* tiles,
           int n_tiles, const int32_t* q_pos, int n_heads, int n_kv_heads, int v_off, int* status,
           cudaStream_t stream, unsigned long long* stamp) {
  using L = AttnSmem<HD>;
  static bool attr = false;
  if (!attr) {
    SPD_CUDA_TRY(cudaFuncSetAttribute(attn_tc_kernel<HD>,
                                      cudaFuncAttributeMaxDynamicSharedMemorySize, int(L::bytes)));
    attr = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf(float(HD));
  SPD_CUDA_TRY(launch_pdl(attn_tc_kernel<HD>, dim3(n_tiles, n_heads), dim3(kThreads), L::bytes,
                          stream, mq, mkv, static_cast<__nv_bfloat16*>(o), ldo, tiles, q_pos,
                          n_heads, n_kv_heads, v_off, scale_log2, status, kWaitBudget, stamp));
  return SPD_OK;
}

// ---- one query per sequence (a decode step) ---------------------------------------------------
// Cluster of kDecSplit CTAs per (tile, head): the tile's single query (its sequence's last position,
// so every key of the sequence is visible) against the keys [first key row, + key count), CTA r of
// the cluster taking the r-th contiguous eighth of them. Within a CTA the 8 warps take keys j with
// j mod 8 = warp; each lane holds HD / 32 consecutive elements of the head. A warp keeps an online
// softmax (running maximum m, sum l, output o) over its keys, four keys' K and V loads in flight;
// the warps' states are merged in warp order, then the CTAs' states in rank order by rank 0
// through distributed shared memory, which writes the output in bf16. At one query per sequence
// there is no tile for the tensor cores to fill: the step reads K and V once, over enough CTAs to
// keep many loads in flight.
constexpr int kDecWarps = 8;
constexpr int kDecSplit = 8;

template <int HD>
__global__ void __launch_bounds__(kDecWarps * 32)
    attn_decode_kernel(const __nv_bfloat16* q, const __nv_bfloat16* kv, int ldkv, int v_off,
                       __nv_bfloat16* __restrict__ o, int ldo, const int4* tiles, int n_heads,
                       int n_kv_heads, float scale_log2, unsigned long long* stamp) {
  constexpr int E = HD / 32;  // elements per lane: 2 or 4
  __shared__ float wm[kDecWarps], wl[kDecWarps];
  __shared__ float wo[kDecWarps][HD];
  __shared__ float cm, cl, co[HD];  // this CTA's merged state
  cg::cluster_group cluster = cg::this_cluster();
  const int rank = int(cluster.block_rank());
  pdl_launch_dependents();
  pdl_wait();
  if (threadIdx.x == 0) stamp_start(stamp);
  const int head = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int4 tl = tiles[blockIdx.x];  // (query row, query count = 1, first key row, key count)
  const int j_lo = rank * tl.w / kDecSplit, j_hi = (rank + 1) * tl.w / kDecSplit;
  const int g = head / (n_heads / n_kv_heads);
  float qv[E];
  {
    const __nv_bfloat16* qp = q + size_t(tl.x) * (n_heads * HD) + head * HD + lane * E;
#pragma unroll
    for (int e = 0; e < E; ++e) qv[e] = __bfloat162float(qp[e]) * scale_log2;
  }
  auto load_row = [&](int j, int off, float (&r)[E]) {
    const __nv_bfloat16* p = kv + size_t(tl.z + j) * ldkv + off + g * HD + lane * E;
    if constexpr (E == 4) {
      const uint2 u = *reinterpret_cast<const uint2*>(p);
      r[0] = __uint_as_float(u.x << 16);
      r[1] = __uint_as_float(u.x & 0xffff0000u);
      r[2] = __uint_as_float(u.y << 16);
      r[3] = __uint_as_float(u.y & 0xffff0000u);
    } else {
      const uint32_t u = *reinterpret_cast<const uint32_t*>(p);
      r[0] = __uint_as_float(u << 16);
      r[1] = __uint_as_float(u & 0xffff0000u);
    }
  };
  float m = -INFINITY, l = 0.0f, acc[E];
#pragma unroll
  for (int e = 0; e < E; ++e) acc[e] = 0.0f;
  for (int j0 = j_lo + warp; j0 < j_hi; j0 += 4 * kDecWarps) {
    float kr[4][E], vr[4][E];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u * kDecWarps;
      if (j < j_hi) {
        load_row(j, 0, kr[u]);
        load_row(j, v_off, vr[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int j = j0 + u * kDecWarps;
      if (j < j_hi) {  // warp-uniform
        float sdot = 0.0f;
#pragma unroll
        for (int e = 0; e < E; ++e) sdot = fmaf(qv[e], kr[u][e], sdot);
#pragma unroll
        for (int off = 16; off; off >>= 1) sdot += __shfl_xor_sync(0xffffffffu, sdot, off);
        const float mn = fmaxf(m, sdot);
        const float corr = exp2f(m - mn), pj = exp2f(sdot - mn);
        l = l * corr + pj;
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = fmaf(pj, vr[u][e], acc[e] * corr);
        m = mn;
      }
    }
  }
  if (lane == 0) {
    wm[warp] = m;
    wl[warp] = l;
  }
#pragma unroll
  for (int e = 0; e < E; ++e) wo[warp][lane * E + e] = acc[e];
  __syncthreads();
  // merge of states (m_i, l_i, o_i): m = max m_i, l = sum l_i 2^(m_i - m), o = sum o_i 2^(m_i - m)
  // (a state without keys has m = -inf and contributes nothing)
  if (threadIdx.x < HD) {
    float mt = -INFINITY;
    for (int w = 0; w < kDecWarps; ++w) mt = fmaxf(mt, wm[w]);
    float lt = 0.0f, ot = 0.0f;
    for (int w = 0; w < kDecWarps; ++w) {
      const float f = wm[w] == -INFINITY ? 0.0f : exp2f(wm[w] - mt);
      lt = fmaf(wl[w], f, lt);
      ot = fmaf(wo[w][threadIdx.x], f, ot);
    }
    co[threadIdx.x] = ot;
    if (threadIdx.x == 0) {
      cm = mt;
      cl = lt;
    }
  }
  cluster.sync();
  if (rank == 0 && threadIdx.x < HD) {
    float ms[kDecSplit], ls[kDecSplit], os[kDecSplit];
#pragma unroll
    for (int r = 0; r < kDecSplit; ++r) {
      ms[r] = *cluster.map_shared_rank(&cm, r);
      ls[r] = *cluster.map_shared_rank(&cl, r);
      os[r] = cluster.map_shared_rank(co, r)[threadIdx.x];
    }
    float mt = -INFINITY;
#pragma unroll
    for (int r = 0; r < kDecSplit; ++r) mt = fmaxf(mt, ms[r]);
    float lt = 0.0f, ot = 0.0f;
#pragma unroll
    for (int r = 0; r < kDecSplit; ++r) {
      const float f = ms[r] == -INFINITY ? 0.0f : exp2f(ms[r] - mt);
      lt = fmaf(ls[r], f, lt);
      ot = fmaf(os[r], f, ot);
    }
    o[size_t(tl.x) * ldo + head * HD + threadIdx.x] = __float2bfloat16_rn(ot / lt);
  }
  cluster.sync();  // the peers' shared memory stays alive until rank 0 has read it
  if (threadIdx.x == 0) stamp_end(stamp);
}

}  // namespace

int attention_run(const void* q, int n_q, const void* kv, int n_kv, int ldkv, int v_off, void* o,
                  int ldo, const int4* tiles, int n_tiles, const int32_t* q_pos, int n_heads,
                  int n_kv_heads, int head_dim, int* status, cudaStream_t stream, double ctx_sum) {
  if (n_tiles <= 0) return SPD_OK;
  if (head_dim != 128 && head_dim != 64)
    return fail(SPD_EUNSUPPORTED, "attention supports head_dim 64 and 128");
  if (n_kv_heads < 1 || n_heads % n_kv_heads)
    return fail(SPD_EINVAL, "n_heads must be a multiple of n_kv_heads");
  if (v_off % 64 || ldkv < v_off + n_kv_heads * head_dim)
    return fail(SPD_EINVAL, "V must start at a multiple of 64 columns inside each K/V row");
  CUtensorMap mq, mkv;
  if (int rc = make_operand_map(&mq, q, n_heads * head_dim, n_q, 128)) return rc;
  if (int rc = make_operand_map(&mkv, kv, ldkv, n_kv, kTK)) return rc;
  // QK^T and PV over each active query's causal context; Q, K, V read once and O written once
  const double fl = 4.0 * head_dim * n_heads * ctx_sum;
  const double by = 2.0 * (2.0 * n_q * n_heads * head_dim + 2.0 * n_kv * n_kv_heads * head_dim);
  unsigned long long* stamp = stamp_slot(TR_ATTN, fl, by);
  const int slot = trace_begin(stream);
  const int rc = (head_dim == 128)
                     ? launch<128>(mq, mkv, o, ldo, tiles, n_tiles, q_pos, n_heads, n_kv_heads,
                                   v_off, status, stream, stamp)
                     : launch<64>(mq, mkv, o, ldo, tiles, n_tiles, q_pos, n_heads, n_kv_heads,
                                  v_off, status, stream, stamp);
  trace_end(slot, stream, TR_ATTN, fl, by);
  return rc;
}

int attention_decode_run(const void* q, const void* kv, int ldkv, int v_off, void* o, int ldo,
                         const int4* tiles, int n_tiles, int n_heads, int n_kv_heads, int head_dim,
                         cudaStream_t stream, double ctx_sum) {
  if (n_tiles <= 0) return SPD_OK;
  if (head_dim != 128 && head_dim != 64)
    return fail(SPD_EUNSUPPORTED, "attention supports head_dim 64 and 128");
  if (n_kv_heads < 1 || n_heads % n_kv_heads)
    return fail(SPD_EINVAL, "n_heads must be a multiple of n_kv_heads");
  if ((ldkv | v_off) % 4) return fail(SPD_EINVAL, "K/V rows must be 8-byte aligned");
  const float scale_log2 = float(1.4426950408889634 / sqrt(double(head_dim)));
  // Q read and O written once per query; K and V of every visible key once per KV head
  const double fl = 4.0 * head_dim * n_heads * ctx_sum;
  const double by = 2.0 * (2.0 * n_tiles * n_heads * head_dim + 2.0 * ctx_sum * n_kv_heads * head_dim);
  unsigned long long* stamp = stamp_slot(TR_ATTN, fl, by);
  const int slot = trace_begin(stream);
  const auto* qb = static_cast<const __nv_bfloat16*>(q);
  const auto* kb = static_cast<const __nv_bfloat16*>(kv);
  auto* ob = static_cast<__nv_bfloat16*>(o);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(n_tiles, n_heads, kDecSplit);
  cfg.blockDim = dim3(kDecWarps * 32);
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 1;
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = kDecSplit;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  if (head_dim == 128)
    SPD_CUDA_TRY(cudaLaunchKernelEx(&cfg, attn_decode_kernel<128>, qb, kb, ldkv, v_off, ob, ldo, tiles,
                                    n_heads, n_kv_heads, scale_log2, stamp));
  else
    SPD_CUDA_TRY(cudaLaunchKernelEx(&cfg, attn_decode_kernel<64>, qb, kb, ldkv, v_off, ob, ldo, tiles,
                                    n_heads, n_kv_heads, scale_log2, stamp));
  trace_end(slot, stream, TR_ATTN, fl, by);
  return SPD_OK;
}

}  // namespace spd
