// tcgen05 bf16 GEMM for the decoder's dense contractions: out = epilogue(X W^T).
//
// Prefill after pruning has few token rows (a few hundred) against large weight matrices, so the
// contraction is weight-stream bound. The WEIGHTS sit on the MMA's M side (128 weight rows per
// tile) and the tokens on its N side (up to 256 per tile): every weight tile is streamed from HBM
// once per token tile.
//
// Two schedules share the kernel:
//  * cluster split-K, when the output has at most half as many tiles as there are SMs: a cluster of
//    C (2, 4 or 8) CTAs owns one output tile, each CTA a contiguous K range. Once every CTA of the
//    cluster has finished its MMAs (its stage ring is idle), each CTA pushes its TMEM accumulator,
//    32-column chunk by chunk, into the ring of the chunk's owner CTA (chunk mod C) with posted
//    distributed-shared-memory stores; after a cluster barrier each owner sums the C copies in rank
//    order from its own shared memory and runs the fused epilogue. No global partials, no remote
//    loads, deterministic.
//  * persistent stream-K otherwise, below.
//
// Persistent stream-K: one CTA per SM. The work is the list of (tile, k-block) units in tile-major
// order; CTA c takes the contiguous units [c U / G, (c+1) U / G). A run of units inside one tile is
// a segment. A segment that covers the whole K range goes straight to the epilogue. Residual (ADD)
// epilogues add into their destination rows with fire-and-forget red.add, whole or split tile
// alike (so the contributions of a split tile land in no fixed order: fp32 rounding may differ in
// the last bits between runs). Other epilogues keep split tiles deterministic: every segment stores
// its fp32 partial in one of its CTA's two slots (head, tail), and the CTA whose segment completes
// the tile's k-block count sums the partials in CTA order and runs the epilogue. No CTA ever waits
// on another.
//
// Stages hold BK = 64 or 128 K elements: one or two weight boxes of 128 rows x 64 (128 B per row
// each, so a 128-wide stage reads 256 contiguous bytes of every weight row) and one or two token
// boxes of the whole token tile x 64. Few large boxes matter: the TMA box rate, not bytes, caps the
// stream when the token tile is cut into small boxes.
//
// Warp roles (320 threads):
//   warp 0 lane 0 : TMA producer  - fills the ring of stages
//   warp 1 lane 0 : MMA issuer    - BK / 16 x tcgen05.mma (K = 16) per stage into one of two TMEM
//                                   accumulators (2 x 256 columns), commit per stage and segment
//   warps 2..9    : epilogue      - two warps per TMEM lane quarter, alternating 32-column chunks;
//                                   tcgen05.ld, fused epilogue; runs on one accumulator while the
//                                   MMA fills the other
#include <cuda_bf16.h>
#include <math.h>
#include <stdio.h>

#include <cooperative_groups.h>

#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace cg = cooperative_groups;

namespace spd {
namespace {

constexpr int kBM = 128;            // weight rows per tile (MMA M)
constexpr int kBK = 64;             // K elements per TMA box (one 128-byte swizzle row)
constexpr int kWBytes = kBM * 128;  // weight box bytes
constexpr int kMaxStages = 8;
constexpr int kSmemPipe = 196608;   // bytes of the stage ring
constexpr int kAccCols = 256;       // TMEM columns per accumulator
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;
constexpr int kCounters = 1 << 16;

struct KArgs {
  int n_out, n_tok, k, tt, n_kb, n_ttiles, units, grid, stages, epi, ldo, rope_rows, head_dim,
      out_cols, kbox, csplit;  // csplit: CTAs per output tile in cluster split-K (1 = stream-K)  // kbox: 64-wide boxes per stage (1 or 2); a k-block is kbox * 64 wide
  void* out;
  const int32_t* rows;
  const uint16_t* bias;
  const int32_t* pos;
  const float2* rope;  // [position][head_dim / 2] (cos, sin)
  float* partial;
  int* counters;
  int* status;
  long long budget;
};

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

// first unit of CTA c, and the CTA that owns unit u, for the balanced split [c U / G, (c+1) U / G)
// (the host guarantees U * (G + 1) < 2^31, so 32-bit arithmetic is exact)
__device__ __forceinline__ int unit_lo(int c, const KArgs& a) { return c * a.units / a.grid; }
__device__ __forceinline__ int cta_of_unit(int u, const KArgs& a) {
  return ((u + 1) * a.grid - 1) / a.units;
}

// Order in which a CTA runs the segments of its unit range [u0, u1): first the partial head
// segment (end of a tile shared with the previous CTA) and the partial tail segment (start of a
// tile shared with the next CTA), then the interior full tiles. The partial tiles' fixups thus run
// early, overlapped with the full tiles' main loop, instead of piling up at the end.
struct SegPlan {
  int u0, u1, n_kb, first_b, last_b, count;
  bool natural, head, tail;
};
__device__ __forceinline__ SegPlan seg_plan(int u0, int u1, int n_kb) {
  SegPlan p;
  p.u0 = u0;
  p.u1 = u1;
  p.n_kb = n_kb;
  p.first_b = ((u0 + n_kb - 1) / n_kb) * n_kb;
  p.last_b = (u1 / n_kb) * n_kb;
  p.natural = p.first_b >= p.last_b;  // no full tile inside: at most two segments, in order
  if (u0 >= u1) {
    p.count = 0;
  } else if (p.natural) {
    const int te = (u0 / n_kb + 1) * n_kb;
    p.count = te < u1 ? 2 : 1;
  } else {
    p.head = u0 < p.first_b;
    p.tail = p.last_b < u1;
    p.count = int(p.head) + int(p.tail) + (p.last_b - p.first_b) / n_kb;
  }
  return p;
}
__device__ __forceinline__ void seg_get(const SegPlan& p, int j, int& s, int& e) {
  if (p.natural) {
    const int te = (p.u0 / p.n_kb + 1) * p.n_kb;
    if (j == 0) {
      s = p.u0;
      e = min(p.u1, te);
    } else {
      s = te;
      e = p.u1;
    }
    return;
  }
  int k = j;
  if (p.head) {
    if (k == 0) {
      s = p.u0;
      e = p.first_b;
      return;
    }
    --k;
  }
  if (p.tail) {
    if (k == 0) {
      s = p.last_b;
      e = p.u1;
      return;
    }
    --k;
  }
  s = p.first_b + k * p.n_kb;
  e = s + p.n_kb;
}

// Applies the epilogue to 32 consecutive tokens t0..t0+31 of weight row n (TMEM lane quarter q).
// trow / tpos: output row and rotary position of each token of the token tile (shared memory,
// indexed from the tile's first token tb).
__device__ __forceinline__ void epilogue_chunk(const KArgs& a, int n, int q, int lane, int w_tile,
                                               int t0, const float (&v)[32], const int* trow,
                                               const int* tpos, int tb) {
  const int nt = a.n_tok;
  switch (a.epi) {
    case EPI_F32:
    case EPI_ADD_F32: {
      if (n >= a.n_out) return;
      float* o = static_cast<float*>(a.out);
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int t = t0 + j;
        if (t < nt) {
          float* p = o + size_t(trow[t - tb]) * a.ldo + n;
          if (a.epi == EPI_ADD_F32) atomicAdd(p, v[j]);  // fire-and-forget red.add
          else *p = v[j];
        }
      }
      return;
    }
    case EPI_BF16:
    case EPI_BIAS_BF16:
    case EPI_BIAS_GELU_BF16: {
      if (n >= a.n_out) return;
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
      const float b = (a.epi == EPI_BF16) ? 0.0f
                                          : __bfloat162float(__ushort_as_bfloat16(a.bias[n]));
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const int t = t0 + j;
        if (t < nt) {
          float x = v[j] + b;
          if (a.epi == EPI_BIAS_GELU_BF16) x = gelu_erf(x);
          o[size_t(trow[t - tb]) * a.ldo + n] = __float2bfloat16_rn(x);
        }
      }
      return;
    }
    case EPI_ROPE_BF16: {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
      if (n < a.rope_rows) {  // tile-uniform: rope_rows is a multiple of 128
        const int hd = a.head_dim, half = hd >> 1;
        const int head = n / hd, g = (n % hd) >> 5;
        const int jf = 16 * g + (lane & 15);
        const int col = head * hd + ((lane < 16) ? jf : half + jf);
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float p = __shfl_xor_sync(0xffffffffu, v[j], 16);
          const int t = t0 + j;
          if (t < nt) {
            const float2 cs = a.rope[size_t(tpos[t - tb]) * half + jf];
            const float y = (lane < 16) ? v[j] * cs.x - p * cs.y : v[j] * cs.x + p * cs.y;
            o[size_t(trow[t - tb]) * a.ldo + col] = __float2bfloat16_rn(y);
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int t = t0 + j;
          if (t < nt) o[size_t(trow[t - tb]) * a.ldo + n] = __float2bfloat16_rn(v[j]);
        }
      }
      return;
    }
    case EPI_SWIGLU_BF16: {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
      const int f = w_tile * 64 + q * 16 + (lane & 15);
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float u = __shfl_xor_sync(0xffffffffu, v[j], 16);
        const int t = t0 + j;
        if (lane < 16 && t < nt && f < a.out_cols) {
          const float g = v[j];
          o[size_t(trow[t - tb]) * a.ldo + f] = __float2bfloat16_rn(g / (1.0f + expf(-g)) * u);
        }
      }
      return;
    }
    default:
      return;
  }
}

__device__ __forceinline__ void epi_bar() {
  asm volatile("bar.sync 1, %0;" ::"n"(kEpiThreads) : "memory");
}
// Barrier over the epilogue warps that returns the OR of `v` over their threads (a uniform result).
__device__ __forceinline__ bool epi_any(bool v) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred p, q;\n\t"
      "setp.ne.u32 p, %1, 0;\n\t"
      "bar.red.or.pred q, 1, %2, p;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(uint32_t(v)), "n"(kEpiThreads)
      : "memory");
  return r != 0;
}

__global__ void __launch_bounds__(kThreads, 1)
    gemm_sk_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_x, const KArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t xbox_bytes = a.tt * 128;
  const uint32_t stage_bytes = a.kbox * (kWBytes + xbox_bytes);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.stages * stage_bytes);
  uint64_t* empty = full + kMaxStages;
  uint64_t* accf = empty + kMaxStages;  // [2] accumulator ready (MMA -> epilogue)
  uint64_t* acce = accf + 2;            // [2] accumulator free  (epilogue -> MMA)
  uint64_t* done = acce + 2;            // MMA drain at teardown
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(done + 1);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] abort [1] last
  volatile int* counts = flags + 2;  // [0] stages issued by TMA, [1] consumed by MMA
  int* trow = const_cast<int*>(counts + 2);  // [256] output row of each token of the tile
  int* tpos = trow + 256;                     // [256] rotary position of each token

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c = blockIdx.x;
  int u0, u1;
  if (a.csplit > 1) {  // cluster split-K: rank r of tile c / C owns k-blocks [r n_kb / C, (r+1) n_kb / C)
    const int tile = c / a.csplit, r = c - tile * a.csplit;
    u0 = tile * a.n_kb + r * a.n_kb / a.csplit;
    u1 = tile * a.n_kb + (r + 1) * a.n_kb / a.csplit;
  } else {
    u0 = unit_lo(c, a);
    u1 = unit_lo(c + 1, a);
  }
  const SegPlan plan = seg_plan(u0, u1, a.n_kb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], kEpiThreads);
    }
    mbar_init(done, 1);
    flags[0] = 0;
    flags[1] = 0;
    counts[0] = 0;
    counts[1] = 0;
    fence_mbar_init();
    prefetch_tmap(&map_w);
    prefetch_tmap(&map_x);
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, 2 * kAccCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  pdl_launch_dependents();
  if (warp == 0) {
    if (lane == 0) {
      // ---- TMA producer ----
      // The first stages' weight boxes do not depend on the previous kernel: they are issued
      // before griddepcontrol.wait, so the weight stream starts while that kernel drains.
      const uint64_t pol_w = policy_evict_first(), pol_x = policy_evict_last();
      int pre_tile[kMaxStages], pre_kb[kMaxStages];
      int n_pre = 0;
      for (int j = 0; j < plan.count && n_pre < a.stages; ++j) {
        int sb, se;
        seg_get(plan, j, sb, se);
        for (int u = sb; u < se && n_pre < a.stages; ++u, ++n_pre) {
          pre_tile[n_pre] = u / a.n_kb;
          pre_kb[n_pre] = u - pre_tile[n_pre] * a.n_kb;
          const int wt = pre_tile[n_pre] / a.n_ttiles;
          uint8_t* st = smem + n_pre * stage_bytes;
          mbar_arrive_expect_tx(&full[n_pre], stage_bytes);
          for (int bx = 0; bx < a.kbox; ++bx)
            tma_load_2d(st + bx * kWBytes, &map_w, &full[n_pre], (pre_kb[n_pre] * a.kbox + bx) * kBK,
                        wt * kBM, pol_w);
        }
      }
      pdl_wait();
      for (int i = 0; i < n_pre; ++i) {
        const int tt_i = pre_tile[i] - (pre_tile[i] / a.n_ttiles) * a.n_ttiles;
        uint8_t* st = smem + i * stage_bytes;
        for (int bx = 0; bx < a.kbox; ++bx)
          tma_load_2d(st + a.kbox * kWBytes + bx * xbox_bytes, &map_x, &full[i],
                      (pre_kb[i] * a.kbox + bx) * kBK, tt_i * a.tt, pol_x);
      }
      counts[0] = n_pre;
      int i = 0;
      bool ok = true;
      for (int j = 0; j < plan.count && ok; ++j) {
        int sb, se;
        seg_get(plan, j, sb, se);
        const int tile = sb / a.n_kb;
        const int wt = tile / a.n_ttiles, tt_i = tile - wt * a.n_ttiles;
        for (int kb = sb - tile * a.n_kb; kb < se - tile * a.n_kb; ++kb, ++i) {
          if (i < n_pre) continue;  // issued above
          const int s = i % a.stages;
          const uint32_t ph = (i / a.stages) & 1;
          if (!mbar_wait(&empty[s], ph ^ 1, flags, a.budget)) {
            flags[0] = 1;
            set_status(a.status, SPD_ETIMEOUT);
            ok = false;
            break;
          }
          uint8_t* st = smem + s * stage_bytes;
          mbar_arrive_expect_tx(&full[s], stage_bytes);
          for (int bx = 0; bx < a.kbox; ++bx) {
            const int kx = (kb * a.kbox + bx) * kBK;
            tma_load_2d(st + bx * kWBytes, &map_w, &full[s], kx, wt * kBM, pol_w);
            tma_load_2d(st + a.kbox * kWBytes + bx * xbox_bytes, &map_x, &full[s], kx, tt_i * a.tt,
                        pol_x);
          }
          counts[0] = i + 1;
        }
      }
    }
  } else if (warp == 1) {
    pdl_wait();
    if (lane == 0) {
      // ---- MMA issuer ----
      const uint32_t idesc = idesc_bf16_f32(kBM, a.tt);
      const int ksub = a.kbox * (kBK / 16);
      int i = 0;
      bool ok = true;
      for (int j = 0; j < plan.count && ok; ++j) {
        int u, seg_end;
        seg_get(plan, j, u, seg_end);
        const int b = j & 1;
        if (!mbar_wait(&acce[b], ((j >> 1) & 1) ^ 1, flags, a.budget)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + b * kAccCols;
        for (int uu = u; uu < seg_end; ++uu, ++i) {
          const int s = i % a.stages;
          const uint32_t ph = (i / a.stages) & 1;
          if (!mbar_wait(&full[s], ph, flags, a.budget)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sw = smem_u32(smem + s * stage_bytes);
          const uint32_t sx = sw + a.kbox * kWBytes;
          for (int kk = 0; kk < ksub; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            mma_bf16(d, sdesc_k128(sw + (kk >> 2) * kWBytes + off),
                     sdesc_k128(sx + (kk >> 2) * xbox_bytes + off), idesc,
                     (uu != u || kk != 0) ? 1u : 0u);
          }
          mma_commit(&empty[s]);
          counts[1] = i + 1;
        }
        if (!ok) break;
        mma_commit(&accf[b]);
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
      }
      mma_commit(done);  // arrives once every MMA issued above has completed
      volatile int no_abort = 0;
      if (!mbar_wait(done, 0, &no_abort, a.budget)) set_status(a.status, SPD_ETIMEOUT);
    }
  } else {
    pdl_wait();
    // ---- epilogue (warps 2..9; warp w reads TMEM lane quarter w % 4, chunk parity (w - 2) / 4) ----
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = q * 32 + lane;
    for (int j = 0; j < plan.count; ++j) {
      int u, seg_end;
      seg_get(plan, j, u, seg_end);
      const int tile = u / a.n_kb;
      const int kb_lo = u - tile * a.n_kb;
      const int seg_len = seg_end - u;
      const int b = j & 1;
      const bool got = mbar_wait(&accf[b], (j >> 1) & 1, flags, a.budget);
      if (epi_any(!got)) {  // every epilogue thread leaves together
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
        break;
      }
      tc_fence_after();
      const int wt = tile / a.n_ttiles, tt_i = tile - wt * a.n_ttiles;
      const int tok0 = tt_i * a.tt;
      const int valid = min(a.tt, a.n_tok - tok0);
      const int n = wt * kBM + row;
      const uint32_t tq = tmem + b * kAccCols + (static_cast<uint32_t>(q * 32) << 16);
      if (a.csplit > 1) break;  // cluster split-K: the accumulator is pushed after the role loops
      // token metadata of this tile, staged once per segment
      const int et = threadIdx.x - 64;
      if (et < valid) {
        trow[et] = a.rows ? a.rows[tok0 + et] : tok0 + et;
        tpos[et] = a.pos ? a.pos[tok0 + et] : 0;
      }
      epi_bar();
      if ((kb_lo == 0 && seg_len == a.n_kb) || a.epi == EPI_ADD_F32) {
        for (int cc = half * 32; cc < valid; cc += 64) {
          float v[32];
          tmem_ld32(tq + cc, v);
          epilogue_chunk(a, n, q, lane, wt, tok0 + cc, v, trow, tpos, tok0);
        }
      } else {
        // deterministic split tile: partial into this CTA's head (0) or tail (1) slot, laid out
        // [32-column chunk][4-column group][128 rows] of float4 (512 contiguous bytes per warp
        // instruction); the last arriver sums the partials in CTA order
        const size_t slot_len = size_t(a.tt / 4) * kBM;
        float4* part = reinterpret_cast<float4*>(a.partial);
        float4* mine = part + size_t(2 * c + (tile == u0 / a.n_kb ? 0 : 1)) * slot_len;
        for (int cc = half * 32; cc < valid; cc += 64) {
          float v[32];
          tmem_ld32(tq + cc, v);
          float4* dst = mine + size_t(cc / 4) * kBM + row;
#pragma unroll
          for (int g = 0; g < 8; ++g)
            __stcg(dst + g * kBM, make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]));
        }
        __threadfence();
        epi_bar();
        if (threadIdx.x == 64) {
          const int old = atomicAdd(&a.counters[tile], seg_len);
          flags[1] = (old + seg_len == a.n_kb);
        }
        epi_bar();
        if (flags[1]) {
          __threadfence();
          const int c_first = cta_of_unit(tile * a.n_kb, a);
          const int c_last = cta_of_unit((tile + 1) * a.n_kb - 1, a);
          for (int cc = half * 32; cc < valid; cc += 64) {
            float v[32], acc[32];
            tmem_ld32(tq + cc, v);
#pragma unroll
            for (int jj = 0; jj < 32; ++jj) acc[jj] = 0.0f;
            // contributors in CTA order, two partial tiles in flight at a time
            for (int o = c_first; o <= c_last; o += 2) {
              float4 x0[8], x1[8];
              const bool l0 = (o != c), l1 = (o + 1 <= c_last) && (o + 1 != c);
              if (l0) {
                const int os = 2 * o + (tile == unit_lo(o, a) / a.n_kb ? 0 : 1);
                const float4* src = part + size_t(os) * slot_len + size_t(cc / 4) * kBM + row;
#pragma unroll
                for (int g = 0; g < 8; ++g) x0[g] = __ldcg(src + g * kBM);
              }
              if (l1) {
                const int os = 2 * (o + 1) + (tile == unit_lo(o + 1, a) / a.n_kb ? 0 : 1);
                const float4* src = part + size_t(os) * slot_len + size_t(cc / 4) * kBM + row;
#pragma unroll
                for (int g = 0; g < 8; ++g) x1[g] = __ldcg(src + g * kBM);
              }
              if (l0) {
#pragma unroll
                for (int g = 0; g < 8; ++g) {
                  acc[4 * g] += x0[g].x;
                  acc[4 * g + 1] += x0[g].y;
                  acc[4 * g + 2] += x0[g].z;
                  acc[4 * g + 3] += x0[g].w;
                }
              } else {
#pragma unroll
                for (int jj = 0; jj < 32; ++jj) acc[jj] += v[jj];
              }
              if (o + 1 <= c_last) {
                if (l1) {
#pragma unroll
                  for (int g = 0; g < 8; ++g) {
                    acc[4 * g] += x1[g].x;
                    acc[4 * g + 1] += x1[g].y;
                    acc[4 * g + 2] += x1[g].z;
                    acc[4 * g + 3] += x1[g].w;
                  }
                } else {
#pragma unroll
                  for (int jj = 0; jj < 32; ++jj) acc[jj] += v[jj];
                }
              }
            }
            epilogue_chunk(a, n, q, lane, wt, tok0 + cc, acc, trow, tpos, tok0);
          }
          if (threadIdx.x == 64) a.counters[tile] = 0;  // ready for the next launch
        }
      }
      epi_bar();  // trow / tpos / flags[1] are reused by the next segment
      tc_fence_before();
      mbar_arrive(&acce[b]);
    }
  }
  __syncthreads();
  if (a.csplit > 1) {
    // cluster reduction: every thread of every CTA of the cluster takes part in both barriers.
    // Receive layout in each owner's ring: [sender][owned chunk][128 rows][36] fp32 (32 columns
    // + 4 of padding: conflict-free 16-byte accesses).
    cg::cluster_group cl = cg::this_cluster();
    const int C = a.csplit, tile = c / C, r = c - tile * C;
    const int wt = tile / a.n_ttiles, tt_i = tile - wt * a.n_ttiles;
    const int tok0 = tt_i * a.tt;
    const int valid = min(a.tt, a.n_tok - tok0);
    const int cpo = (a.tt / 32 + C - 1) / C;  // chunks owned per CTA
    float* recv = reinterpret_cast<float*>(smem);
    const int et = threadIdx.x - 64;
    if (et >= 0 && et < valid) {
      trow[et] = a.rows ? a.rows[tok0 + et] : tok0 + et;
      tpos[et] = a.pos ? a.pos[tok0 + et] : 0;
    }
    cl.sync();  // every ring of the cluster is idle
    if (warp >= 2 && !flags[0]) {
      const int q = warp & 3, half = (warp - 2) >> 2, row = q * 32 + lane;
      tc_fence_after();
      const uint32_t tq = tmem + (static_cast<uint32_t>(q * 32) << 16);
      for (int ci = half; ci * 32 < valid; ci += 2) {
        float v[32];
        tmem_ld32(tq + ci * 32, v);
        const int owner = ci % C, lc = ci / C;
        const uint32_t dst =
            dsmem_addr(recv + (size_t(r * cpo + lc) * kBM + row) * 36, uint32_t(owner));
#pragma unroll
        for (int g = 0; g < 8; ++g)
          st_dsmem_v4(dst + g * 16, make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]));
      }
    }
    cl.sync();  // all pushes have landed
    if (warp >= 2 && !flags[0]) {
      const int q = warp & 3, half = (warp - 2) >> 2, row = q * 32 + lane;
      const int n = wt * kBM + row;
      for (int lc = half; lc < cpo; lc += 2) {
        const int ci = r + lc * C;
        if (ci * 32 >= valid) break;
        float acc[32];
#pragma unroll
        for (int jj = 0; jj < 32; ++jj) acc[jj] = 0.0f;
        for (int sdr = 0; sdr < C; ++sdr) {
          const float4* src =
              reinterpret_cast<const float4*>(recv + (size_t(sdr * cpo + lc) * kBM + row) * 36);
#pragma unroll
          for (int g = 0; g < 8; ++g) {
            const float4 x = src[g];
            acc[4 * g] += x.x;
            acc[4 * g + 1] += x.y;
            acc[4 * g + 2] += x.z;
            acc[4 * g + 3] += x.w;
          }
        }
        epilogue_chunk(a, n, q, lane, wt, tok0 + ci * 32, acc, trow, tpos, tok0);
      }
    }
  }
  if (threadIdx.x == 0 && flags[0]) {
    // drain: TMA loads issued but never consumed must land before the CTA exits
    for (int i = counts[1]; i < counts[0]; ++i) {
      volatile int no_abort = 0;
      mbar_wait(&full[i % a.stages], (i / a.stages) & 1, &no_abort, a.budget);
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 0) tmem_dealloc(tmem, 2 * kAccCols);
}

// ---- host side -------------------------------------------------------------------------------
using EncodeFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                              const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                              CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                              CUtensorMapFloatOOBfill);

EncodeFn encode_fn() {
  static EncodeFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeFn>(p);
  });
  return fn;
}

int make_map(CUtensorMap* map, const void* ptr, int inner, int outer, int box_outer) {
  EncodeFn fn = encode_fn();
  if (!fn) return fail(SPD_ECUDA, "cuTensorMapEncodeTiled unavailable");
  if ((reinterpret_cast<uintptr_t>(ptr) & 15) || (inner % 8))
    return fail(SPD_EINVAL, "GEMM operand must be 16-byte aligned with K a multiple of 8");
  cuuint64_t dims[2] = {cuuint64_t(inner), cuuint64_t(outer)};
  cuuint64_t strides[1] = {cuuint64_t(inner) * 2};
  cuuint32_t box[2] = {kBK, cuuint32_t(box_outer)};
  cuuint32_t estr[2] = {1, 1};
  CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides,
                  box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS) return fail(SPD_ECUDA, "cuTensorMapEncodeTiled failed (%d)", int(r));
  return SPD_OK;
}

}  // namespace

size_t gemm_scratch_bytes() { return kGemmSlotFloats * sizeof(float) + kCounters * sizeof(int) + 512; }

int make_weight_map(CUtensorMap* map, const void* w, int n_out, int k) {
  return make_map(map, w, k, n_out, kBM);
}

int gemm_run(const GemmProblem& p, const GemmScratch& s, cudaStream_t stream) {
  if (p.n_tok <= 0 || p.n_out <= 0) return SPD_OK;
  if (p.k <= 0) return fail(SPD_EINVAL, "GEMM K must be positive");
  CUtensorMap map_w, map_x;
  if (p.map_w) {
    map_w = *p.map_w;
  } else if (int rc = make_map(&map_w, p.w, p.k, p.n_out, kBM)) {
    return rc;
  }
  KArgs a{};
  a.n_out = p.n_out;
  a.n_tok = p.n_tok;
  a.k = p.k;
  a.n_ttiles = (p.n_tok + 255) / 256;
  a.tt = ((p.n_tok + a.n_ttiles - 1) / a.n_ttiles + 31) / 32 * 32;
  if (int rc = make_map(&map_x, p.x, p.k, p.n_tok, a.tt)) return rc;
  // 128-wide k-blocks when at least two fit in the ring (two 128-byte runs per weight row)
  a.kbox = (2 * 2 * (kWBytes + a.tt * 128) <= kSmemPipe && p.k > kBK) ? 2 : 1;
  a.n_kb = (p.k + a.kbox * kBK - 1) / (a.kbox * kBK);
  const int n_wtiles = (p.n_out + kBM - 1) / kBM;
  const long long tiles = (long long)n_wtiles * a.n_ttiles;
  if (tiles > s.n_counters) return fail(SPD_EUNSUPPORTED, "GEMM has too many output tiles");
  const long long units = tiles * a.n_kb;
  if (units > 0x3fffffffLL) return fail(SPD_EUNSUPPORTED, "GEMM too large");
  a.units = int(units);
  const int sms = num_sms();
  const int stage_bytes = a.kbox * (kWBytes + a.tt * 128);
  a.stages = kSmemPipe / stage_bytes;
  if (a.stages > kMaxStages) a.stages = kMaxStages;
  // cluster split-K when the tiles fill at most half the SMs: C CTAs per tile (each >= 1 k-block)
  a.csplit = 1;
  if (tiles * 2 <= sms) {
    int C = 2;
    while (C < 8 && tiles * C * 2 <= sms && C * 2 <= a.n_kb) C *= 2;
    // the ring receives C copies of each CTA's share of 32-column chunks ([128][36] fp32 each)
    const int chunks = a.tt / 32, cpo = (chunks + C - 1) / C;
    const size_t recv = size_t(C) * cpo * kBM * 36 * sizeof(float);
    if (C <= a.n_kb && recv <= size_t(a.stages) * stage_bytes) a.csplit = C;
  }
  // one CTA per SM with at least 2 units each; every CTA owns two partial slots (head, tail)
  long long grid = sms;
  if (grid > (units + 1) / 2) grid = (units + 1) / 2;
  const size_t per_slot = size_t(a.tt) * kBM;
  if (size_t(2 * grid) * per_slot > s.partial_floats) grid = s.partial_floats / (2 * per_slot);
  if (grid < 1) grid = 1;
  if (units * (grid + 1) >= (1LL << 31)) return fail(SPD_EUNSUPPORTED, "GEMM too large");
  if (a.csplit > 1) grid = tiles * a.csplit;
  a.grid = int(grid);
  a.epi = p.epi;
  a.out = p.out;
  a.ldo = p.ldo;
  a.rows = p.rows;
  a.bias = p.bias;
  a.pos = p.pos;
  a.rope = reinterpret_cast<const float2*>(p.rope);
  a.rope_rows = p.rope_rows;
  a.head_dim = p.head_dim;
  a.out_cols = p.out_cols;
  a.partial = s.partial;
  a.counters = s.counters;
  a.status = s.status;
  a.budget = kWaitBudget;

  const size_t smem = size_t(a.stages) * stage_bytes + 1024 + 256 + 2048;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(gemm_sk_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kSmemPipe + 1024 + 256 + 16384);
  });
  if (attr_err != cudaSuccess)
    return fail(SPD_ECUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(attr_err));
  const int slot = trace_begin(stream);
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(a.grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = a.csplit;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    SPD_CUDA_TRY(cudaLaunchKernelEx(&cfg, gemm_sk_kernel, map_w, map_x, a));
  }
  if (slot >= 0) {
    // algorithmic work: valid output columns only; weights, activations and results move once
    const double cols = (p.epi == EPI_SWIGLU_BF16) ? 2.0 * p.out_cols : double(p.n_out);
    const double out_cols = (p.epi == EPI_SWIGLU_BF16) ? double(p.out_cols) : double(p.n_out);
    const double ob = (p.epi == EPI_F32) ? 4.0 : (p.epi == EPI_ADD_F32) ? 8.0 : 2.0;
    trace_end(slot, stream, TR_GEMM, 2.0 * p.n_tok * cols * p.k,
              2.0 * cols * p.k + 2.0 * p.n_tok * p.k + ob * p.n_tok * out_cols);
  }
  return SPD_OK;
}

}  // namespace spd
