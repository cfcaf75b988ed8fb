// tcgen05 bf16 GEMM for the decoder's dense contractions: out = epilogue(X W^T).
//
// Prefill after pruning has few token rows (a few hundred) against large weight matrices, so the
// contraction is weight-stream bound. The WEIGHTS sit on the MMA's M side and the tokens on its N
// side (up to 256 per tile): every weight tile is streamed from HBM once per token tile. A tile is
// 128 weight rows, or 256 (two M = 128 MMAs sharing each token box) when the token tile is at most
// 64 wide and the stages would otherwise carry few weight bytes.
//
// Two schedules share the kernel:
//  * cluster split-K, when the output has at most half as many tiles as there are SMs: a cluster of
//    C (2, 4 or 8) CTAs owns one output tile, each CTA a contiguous K range. Once every CTA of the
//    cluster has finished its MMAs (its stage ring is idle), each CTA pushes one 128-row half of its
//    TMEM accumulator, 32-column chunk by chunk, into the ring of the chunk's owner CTA (chunk mod
//    C) with posted distributed-shared-memory stores; after a cluster barrier each owner sums the C
//    copies in rank order from its own shared memory and runs the fused epilogue; then the second
//    half. No global partials, no remote loads, deterministic.
//    Residual (ADD) epilogues split K the same way without a cluster: each CTA adds its partial
//    into the destination rows with red.add, which the residual update does anyway.
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
// Stages hold BK = 64 or 128 K elements: one or two weight boxes of 128 nh rows x 64 (a 128-wide
// stage reads 256 contiguous bytes of every weight row) and one or two token boxes of the whole
// token tile x 64. Few large boxes matter: the TMA box rate, not bytes, caps the stream when a tile
// is cut into small boxes.
//
// The kernel is instantiated once per epilogue, and every epilogue works on 8 accumulator columns
// at a time (tcgen05.ld x8, a rolled loop around an 8-wide body): with all epilogues inlined and
// unrolled over 32 columns the code outgrew the instruction cache and the epilogue ran several
// times slower than its arithmetic and stores.
//
// Warp roles (320 threads):
//   warp 0 lane 0 : TMA producer  - fills the ring of stages
//   warp 1 lane 0 : MMA issuer    - nh x BK / 16 tcgen05.mma (M = 128, K = 16) per stage into the
//                                   128-row halves of a TMEM accumulator; commit per stage and per
//                                   segment. Two accumulators fit in the 512 TMEM columns unless
//                                   nh = 2 with a token tile wider than 128 (the epilogue drains
//                                   one while the MMA fills the other).
//   warps 2..9    : epilogue      - two warps per TMEM lane quarter, alternating 8-column groups;
//                                   tcgen05.ld, fused epilogue
#include <cuda_bf16.h>
#include <math.h>
#include <stdio.h>

#include <cooperative_groups.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace cg = cooperative_groups;

namespace spd {
namespace {

constexpr int kBM = 128;            // weight rows per MMA (M) and per TMEM lane set
constexpr int kBK = 64;             // K elements per box (one 128-byte swizzle row)
constexpr int kHalfW = kBM * 128;   // bytes of 128 weight rows x 64
constexpr int kMaxStages = 8;
constexpr int kSmemPipe = 196608;   // bytes of the stage ring
constexpr int kAccCols = 256;       // TMEM columns per accumulator buffer (double-buffered tiles)
constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;
constexpr int kCounters = 1 << 16;
constexpr int kRecvPitch = 36;      // fp32 per row of a received 32-column chunk (conflict-free)

struct KArgs {
  int n_out, n_tok, k, tt, n_kb, n_ttiles, units, grid, stages, ldo, rope_rows, head_dim,
      out_cols, kbox, csplit, cluster, nbuf, hoff, nh, ldo2, split, accs;
  // kbox: 64-wide boxes per stage (1 or 2); a k-block is kbox * 64 wide
  // csplit: CTAs per output tile in split-K (1 = stream-K); cluster: split-K CTAs reduce through
  // distributed shared memory (0: ADD epilogue, every CTA adds its own partial)
  // nbuf: TMEM accumulator buffers; hoff: TMEM column offset of the second 128-row half
  // nh: 128-row halves per tile (1 or 2); accs: TMEM columns between accumulator buffers
  // CTA-pair kernels: a work item (grid entry) is a pair of CTAs sharing one M = 256 tile
  void* out;
  void* out2;
  const int32_t* rows;
  const int32_t* rows2;  // EPI_QKV_BF16: row of token t in out2 (null = t)
  const uint16_t* bias;
  const int32_t* pos;
  const float2* rope;  // [head_dim / 2] rotary frequency theta^(-2j / head_dim) as fp32 (hi, lo)
  float* partial;
  int* counters;
  int* status;
  long long budget;
  int determ;                 // deterministic mode: every output element summed in a fixed order
  int dpr, rem_tiles, whole;  // data-parallel + remainder schedule (seg_plan_dpr)
  float* acc;                 // dpr: fp32 accumulation buffers of the remainder tiles (zero at start)
  int vec_red;  // residual epilogue: 16-byte reductions (n_out, ldo multiples of 4, out aligned)
  int staged;  // rotary epilogues: the last whole segment of a CTA goes out through shared memory
  const float* norm_h;  // matrix-vector path: input RMSNorm (see GemmProblem)
  const uint16_t* norm_gain;
  const int32_t* norm_rows;
  float norm_eps;
  unsigned long long* stamp;  // launch stamp [start, end] (measurement; null = off)
};

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  return v;
}

// 4 x 4 transposes inside each lane quad of a warp: lane k of a quad holds values v[j] of row n0 + k
// (n0 = 4 (lane / 4)) for columns j = 0..7; afterwards w[4 b + c] = value of row n0 + c, column
// 4 b + k (b = 0, 1), so that the lane owns four consecutive rows of two columns.
__device__ __forceinline__ void quad_transpose8(const float (&v)[8], float (&w)[8], int lane) {
#pragma unroll
  for (int j = 0; j < 8; ++j) w[j] = v[j];
  const int k = lane & 3;
#pragma unroll
  for (int bit = 0; bit < 2; ++bit) {
    const int m = 1 << bit;
    const bool hi = (k >> bit) & 1;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      if (j & m) continue;
      const float send = hi ? w[j] : w[j + m];
      const float recv = __shfl_xor_sync(0xffffffffu, send, m);
      if (hi) w[j] = recv;
      else w[j + m] = recv;
    }
  }
}

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
  bool dpr;                     // data-parallel + remainder schedule (seg_plan_dpr)
  int n_rsegs, whole0, n_whole;
};
__device__ __forceinline__ SegPlan seg_plan(int u0, int u1, int n_kb) {
  SegPlan p{};
  p.dpr = false;
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
// Data-parallel + remainder schedule: the first rem_tiles tiles are split in K over the work items,
// each remainder tile over a contiguous group of G / rem_tiles items (G the work items) so that no
// item holds parts of two remainder tiles (a second remainder segment would wait for the first
// one's accumulator to drain); the contributions of a remainder tile meet in an fp32 accumulation
// buffer at L2. Then the item runs the whole tiles rem_tiles + wc W .. + W - 1, which need no
// fixup. The remainder comes first, so its fixups overlap the whole tiles' main loops.
__device__ __forceinline__ SegPlan seg_plan_dpr(int wc, int grid, int rem_tiles, int whole, int n_kb) {
  SegPlan p{};
  p.dpr = true;
  p.n_kb = n_kb;
  int rt = int((long long)wc * rem_tiles / grid);  // this item's remainder tile
  while (rt + 1 < rem_tiles && (long long)(rt + 1) * grid / rem_tiles <= wc) ++rt;
  while (rt > 0 && (long long)rt * grid / rem_tiles > wc) --rt;
  const int g0 = int((long long)rt * grid / rem_tiles);
  const int ng = int((long long)(rt + 1) * grid / rem_tiles) - g0, li = wc - g0;
  p.u0 = rt * n_kb + li * n_kb / ng;
  p.u1 = rt * n_kb + (li + 1) * n_kb / ng;
  p.n_rsegs = p.u0 < p.u1 ? 1 : 0;
  p.whole0 = rem_tiles + wc * whole;
  p.n_whole = whole;
  p.count = p.n_rsegs + p.n_whole;
  return p;
}
__device__ __forceinline__ void seg_get(const SegPlan& p, int j, int& s, int& e) {
  if (p.dpr) {
    if (j < p.n_rsegs) {
      const int t = p.u0 / p.n_kb + j;
      s = max(p.u0, t * p.n_kb);
      e = min(p.u1, (t + 1) * p.n_kb);
    } else {
      s = (p.whole0 + j - p.n_rsegs) * p.n_kb;
      e = s + p.n_kb;
    }
    return;
  }
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

// 2 pi = kTwoPiHi + kTwoPiLo; kTwoPiHi = 6.28125 has 8 significant bits, so k kTwoPiHi is exact
// in fp32 for |k| < 2^16 (two-constant Cody-Waite reduction).
constexpr float kTwoPiHi = 6.28125f;
constexpr float kTwoPiLo = 1.9353071795864769e-3f;
constexpr float kInvTwoPi = 0.15915494309189535f;

// cos and sin of position p times frequency (f.x + f.y). The product is formed exactly (two-product)
// and reduced to about [-pi, pi] with the split 2 pi above, so the angle is within ~2e-7 of exact
// for angles below 2^16 x 2 pi; __sincosf then adds at most 2^-21.4.
__device__ __forceinline__ void rope_cos_sin(int p, float2 f, float& c, float& sn) {
  const float pf = float(p);  // exact for p < 2^24
  const float x_hi = pf * f.x;
  const float x_lo = fmaf(pf, f.x, -x_hi) + pf * f.y;
  const float k = rintf(x_hi * kInvTwoPi);
  float r = fmaf(-k, kTwoPiHi, x_hi);  // exact
  r = fmaf(-k, kTwoPiLo, r) + x_lo;
  __sincosf(r, &sn, &c);
}

// Rotary embedding of weight row nn (rows laid out in rotary pairs: lane l < 16 of a 32-row group
// holds pair element j, lane l + 16 element j + head_dim / 2) for 8 tokens t0 + j, handed to
// store(j, col, value) with col = head * head_dim + rotated index. The angles are computed in
// registers: a per-position table would cost an L2 round trip per 8 tokens.
// The angles of rope8: lanes l and l + 16 rotate by the same angles, so each evaluates those of four
// of the 8 tokens t0 + j (lane l the first four, lane l + 16 the last four) and they trade them;
// pos_of(t) is the rotary position of token t.
template <typename PosOf>
__device__ __forceinline__ void rope_angles4(const KArgs& a, int nn, int lane, int t0, PosOf pos_of,
                                             float (&cm)[4], float (&sm)[4]) {
  const int nt = a.n_tok;
  const int jf = 16 * ((nn % a.head_dim) >> 5) + (lane & 15);
  const float2 fr = a.rope[jf];
  const int hi = lane >> 4;
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int t = min(t0 + 4 * hi + i, nt - 1);
    rope_cos_sin(pos_of(t), fr, cm[i], sm[i]);
  }
}

// rope8 with this lane's four angles given (cm, sm as computed by rope_angles4).
template <typename Store>
__device__ __forceinline__ void rope8_rot(const KArgs& a, int nn, int lane, const float (&v)[8],
                                          const float (&cm)[4], const float (&sm)[4], Store store) {
  const int hd = a.head_dim, half = hd >> 1;
  const int head = nn / hd, g = (nn % hd) >> 5;
  const int jf = 16 * g + (lane & 15);
  const int col = head * hd + ((lane < 16) ? jf : half + jf);
  const float sgn = (lane < 16) ? -1.0f : 1.0f;
  const int hi = lane >> 4;
  float y[8];
#pragma unroll
  for (int i = 0; i < 4; ++i) {  // branch-free math, then the stores
    const float co = __shfl_xor_sync(0xffffffffu, cm[i], 16);
    const float so = __shfl_xor_sync(0xffffffffu, sm[i], 16);
    const float c_lo = hi ? co : cm[i], s_lo = hi ? so : sm[i];  // token i
    const float c_hi = hi ? cm[i] : co, s_hi = hi ? sm[i] : so;  // token i + 4
    const float p_lo = __shfl_xor_sync(0xffffffffu, v[i], 16);
    const float p_hi = __shfl_xor_sync(0xffffffffu, v[i + 4], 16);
    y[i] = fmaf(sgn * p_lo, s_lo, v[i] * c_lo);
    y[i + 4] = fmaf(sgn * p_hi, s_hi, v[i + 4] * c_hi);
  }
#pragma unroll
  for (int j = 0; j < 8; ++j) store(j, col, y[j]);
}

template <typename Store>
__device__ __forceinline__ void rope8(const KArgs& a, int nn, int lane, int t0, const float (&v)[8],
                                      const int* tpos, int tb, Store store) {
  float cm[4], sm[4];
  rope_angles4(a, nn, lane, t0, [&](int t) { return tpos[t - tb]; }, cm, sm);
  rope8_rot(a, nn, lane, v, cm, sm, store);
}

// rope8 stored as bf16 to row row_of(t) of o (skipped when negative or past the tokens).
template <typename RowOf>
__device__ __forceinline__ void rope_store8(const KArgs& a, __nv_bfloat16* o, int ldo, int nn,
                                            int lane, int t0, const float (&v)[8], const int* tpos,
                                            int tb, RowOf row_of) {
  const int nt = a.n_tok;
  rope8(a, nn, lane, t0, v, tpos, tb, [&](int j, int col, float y) {
    const int t = t0 + j;
    const int r = (t < nt) ? row_of(t) : -1;
    if (r >= 0) o[size_t(r) * ldo + col] = __float2bfloat16_rn(y);
  });
}

// Staged output of the rotary epilogues: the CTA's 128-column block of the output for 8 tokens,
// written as bf16 into shared memory rows of kStgPitch bytes (token t0 + j - tb at row t0 + j -
// tb, column col - c0) and copied out row by row afterwards (stage_copy_out).
constexpr int kStgPitch = 256;
template <int EPI>
__device__ __forceinline__ void stage8(const KArgs& a, int n, int lane, int t0, const float (&v)[8],
                                       const int* tpos, int tb, uint8_t* stg,
                                       const float* cs = nullptr) {
  const bool second = EPI == EPI_QKV_BF16 && n >= a.split;  // a K/V row of the fused QKV GEMM
  const int nn = second ? n - a.split : n;                   // row within its output
  const int c0 = nn & ~127;
  uint8_t* base = stg + size_t(t0 - tb) * kStgPitch;
  auto put = [&](int j, int col, float y) {
    *reinterpret_cast<__nv_bfloat16*>(base + j * kStgPitch + 2 * (col - c0)) = __float2bfloat16_rn(y);
  };
  if ((EPI == EPI_QKV_BF16 && !second) || nn < a.rope_rows) {  // warp-uniform
    if (cs) {  // the angles from the rotary table: (cos, sin) of the lane's four tokens
      const float cm[4] = {cs[0], cs[2], cs[4], cs[6]}, sm[4] = {cs[1], cs[3], cs[5], cs[7]};
      rope8_rot(a, nn, lane, v, cm, sm, put);
    } else {
      rope8(a, nn, lane, t0, v, tpos, tb, put);
    }
  } else {
#pragma unroll
    for (int j = 0; j < 8; ++j) put(j, nn, v[j]);
  }
}

// Copies the staged 128-column block of weight rows [n0, n0 + 128) out to global memory: one
// 256-byte bulk copy per token row, issued by epilogue thread et for token tok0 + et (skipped past
// the valid tokens and for negative rows). Every epilogue thread waits for its copies to complete.
template <int EPI>
__device__ __forceinline__ void stage_copy_out(const KArgs& a, int n0, int et, int tok0, int valid,
                                               const int* trow, const uint8_t* stg) {
  if (et < valid) {
    const bool second = EPI == EPI_QKV_BF16 && n0 >= a.split;
    const int nn0 = second ? n0 - a.split : n0;
    const int t = tok0 + et;
    const int r = second ? (a.rows2 ? a.rows2[t] : t) : trow[et];
    if (r >= 0) {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(second ? a.out2 : a.out);
      const int ldo = second ? a.ldo2 : a.ldo;
      bulk_store(o + size_t(r) * ldo + nn0, stg + size_t(et) * kStgPitch, kStgPitch);
    }
  }
  bulk_commit();
  bulk_wait_all();
}

// Applies epilogue EPI to 8 consecutive tokens t0..t0+7 of weight row n (TMEM lane quarter q;
// w_tile = the 128-row block n / 128). trow / tpos: output row and rotary position of each token
// of the token tile (shared memory, indexed from the tile's first token tb). Warp-uniform calls.
template <int EPI>
__device__ __forceinline__ void epilogue8(const KArgs& a, int n, int q, int lane, int w_tile,
                                          int t0, const float (&v)[8], const int* trow,
                                          const int* tpos, int tb) {
  const int nt = a.n_tok;
  if constexpr (EPI == EPI_ADD_F32) {
    if (a.vec_red && !a.determ) {
      // 4 x 4 transposes inside each lane quad: lane k of a quad holds columns c0 .. c0 + 3 (c0 =
      // n rounded down to 4) of tokens t0 + k and t0 + 4 + k afterwards, added with two 16-byte
      // reductions instead of eight 4-byte ones (the residual update is bound by L2 atomics)
      float w[8];
      quad_transpose8(v, w, lane);
      const int k = lane & 3;
      const int c0 = n & ~3;
      if (c0 < a.n_out) {  // n_out is a multiple of 4: a quad is in or out as a whole
        float* o = static_cast<float*>(a.out);
#pragma unroll
        for (int blk = 0; blk < 2; ++blk) {
          const int t = t0 + 4 * blk + k;
          const int r = t < nt ? trow[t - tb] : -1;  // negative: a padding row of a device list
          if (r >= 0) red_add_v4(o + size_t(r) * a.ldo + c0, w[4 * blk], w[4 * blk + 1],
                                 w[4 * blk + 2], w[4 * blk + 3]);
        }
      }
      return;
    }
  }
  if constexpr (EPI == EPI_F32 || EPI == EPI_ADD_F32) {
    if (n >= a.n_out) return;
    float* o = static_cast<float*>(a.out);
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int t = t0 + j;
      const int r = t < nt ? trow[t - tb] : -1;  // negative: a padding row of a device-built list
      if (r >= 0) {
        float* p = o + size_t(r) * a.ldo + n;
        if constexpr (EPI == EPI_ADD_F32) {
          if (a.determ) *p += v[j];  // the tile's one finalizer: a plain read-modify-write
          else atomicAdd(p, v[j]);   // fire-and-forget red.add
        }
        else *p = v[j];
      }
    }
  } else if constexpr (EPI == EPI_BF16 || EPI == EPI_BIAS_BF16 || EPI == EPI_BIAS_GELU_BF16) {
    if (n >= a.n_out) return;
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
    const float b =
        (EPI == EPI_BF16) ? 0.0f : __bfloat162float(__ushort_as_bfloat16(a.bias[n]));
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int t = t0 + j;
      if (t < nt) {
        float x = v[j] + b;
        if constexpr (EPI == EPI_BIAS_GELU_BF16) x = gelu_erf(x);
        o[size_t(trow[t - tb]) * a.ldo + n] = __float2bfloat16_rn(x);
      }
    }
  } else if constexpr (EPI == EPI_ROPE_BF16) {
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
    if (n < a.rope_rows) {  // warp-uniform: rope_rows is a multiple of 32
      rope_store8(a, o, a.ldo, n, lane, t0, v, tpos, tb, [&](int t) { return trow[t - tb]; });
    } else if (n < a.n_out) {
#pragma unroll
      for (int j = 0; j < 8; ++j) {
        const int t = t0 + j;
        if (t < nt) o[size_t(trow[t - tb]) * a.ldo + n] = __float2bfloat16_rn(v[j]);
      }
    }
  } else if constexpr (EPI == EPI_QKV_BF16) {
    if (n < a.split) {  // query rows (warp-uniform: split is a multiple of 128)
      rope_store8(a, static_cast<__nv_bfloat16*>(a.out), a.ldo, n, lane, t0, v, tpos, tb,
                  [&](int t) { return trow[t - tb]; });
    } else {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out2);
      const int nn = n - a.split;
      if (nn < a.rope_rows) {
        rope_store8(a, o, a.ldo2, nn, lane, t0, v, tpos, tb,
                    [&](int t) { return a.rows2 ? a.rows2[t] : t; });
      } else if (n < a.n_out) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
          const int t = t0 + j;
          if (t < nt) o[size_t(a.rows2 ? a.rows2[t] : t) * a.ldo2 + nn] = __float2bfloat16_rn(v[j]);
        }
      }
    }
  } else if constexpr (EPI == EPI_LSE_F32) {
    // the statistics of this warp's 32 weight rows (vocabulary words) for each of the 8 tokens:
    // warp max, then the sums of e^(z - m) and e^(z - m) (z - m); lane j stores token t0 + j's
    float m8[8], s8[8], u8[8];
    const bool live = n < a.n_out;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      float m = live ? v[j] : -INFINITY;
#pragma unroll
      for (int off = 16; off; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
      const float d = live ? v[j] - m : 0.0f;
      const float e = live ? __expf(d) : 0.0f;
      float sj = e, uj = e * d;
#pragma unroll
      for (int off = 16; off; off >>= 1) {
        sj += __shfl_xor_sync(0xffffffffu, sj, off);
        uj += __shfl_xor_sync(0xffffffffu, uj, off);
      }
      m8[j] = m;
      s8[j] = sj;
      u8[j] = uj;
    }
    float4* o = static_cast<float4*>(a.out);
    const int g = n >> 5;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int t = t0 + j;
      if (lane == j && t < nt) o[size_t(t) * a.ldo + g] = make_float4(m8[j], s8[j], u8[j], 0.0f);
    }
  } else if constexpr (EPI == EPI_SWIGLU_BF16) {
    // lanes l and l + 16 hold gate and up of the same FFN channel f: after one exchange lane l
    // finishes the even tokens of the group and lane l + 16 the odd ones
    __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
    const int f = w_tile * 64 + q * 16 + (lane & 15);
    const int odd = lane >> 4;
    float y[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      // lane < 16 sends v[2i + 1] (its gate of the odd token) and receives the up of the even one
      const float e0 = v[2 * i], e1 = v[2 * i + 1];
      const float mine = odd ? e1 : e0, other = odd ? e0 : e1;
      const float recv = __shfl_xor_sync(0xffffffffu, other, 16);
      const float g = odd ? recv : mine, u = odd ? mine : recv;
      y[i] = __fdividef(g, 1.0f + __expf(-g)) * u;  // SiLU(g) u; 0 once 1 + e^-g passes 2^126
    }
    if (f < a.out_cols) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int t = t0 + 2 * i + odd;
        if (t < nt) o[size_t(trow[t - tb]) * a.ldo + f] = __float2bfloat16_rn(y[i]);
      }
    }
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

__device__ __forceinline__ void add4(float (&acc)[8], int o, const float4& x) {
  acc[o] += x.x;
  acc[o + 1] += x.y;
  acc[o + 2] += x.z;
  acc[o + 3] += x.w;
}

// 10 warps: three share an SM sub-partition's 16K registers, so at most 168 registers a thread.
// PAIR: a cluster of two CTAs computes 256 weight rows x the token tile with M = 256 MMAs
// (tcgen05 cta_group::2): each CTA loads its own 128 weight rows and half of the tokens, the
// even CTA issues the MMAs, each CTA's TMEM holds its 128 rows. Per weight byte that moves 5
// bytes through shared memory instead of 6 (the token half is read by both tensor cores but
// written once), the limit of the single-CTA main loop.
// DET (residual epilogue only): deterministic mode, split tiles through the ordered partial slots
// and plain read-modify-writes instead of red.add (a separate instance: the slot fixups would raise
// the register count of the red.add instance, and with it the registers a co-resident kernel of the
// programmatic launch chain can get).
template <int EPI, bool PAIR, bool DET = false>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_sk_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_x, const KArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t xbox_bytes = (PAIR ? a.tt / 2 : a.tt) * 128;
  const uint32_t wbox_bytes = a.nh * kHalfW;
  const uint32_t stage_bytes = a.kbox * (wbox_bytes + xbox_bytes);
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
  const int c = blockIdx.x;              // CTA index (partial slots)
  const int wc = PAIR ? c >> 1 : c;      // work item
  const int prank = PAIR ? c & 1 : 0;    // CTA within the pair (cluster rank); 0 issues the MMAs
  int u0, u1;
  if (a.csplit > 1) {  // split-K: rank r of tile wc / C owns k-blocks [r n_kb / C, (r+1) n_kb / C)
    const int tile = wc / a.csplit, r = wc - tile * a.csplit;
    u0 = tile * a.n_kb + r * a.n_kb / a.csplit;
    u1 = tile * a.n_kb + (r + 1) * a.n_kb / a.csplit;
  } else {
    u0 = unit_lo(wc, a);
    u1 = unit_lo(wc + 1, a);
  }
  const SegPlan plan = a.dpr ? seg_plan_dpr(wc, a.grid, a.rem_tiles, a.whole, a.n_kb)
                             : seg_plan(u0, u1, a.n_kb);

  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&accf[b], 1);
      mbar_init(&acce[b], PAIR ? 2 : kEpiThreads);  // PAIR: one arrive per CTA
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
    if constexpr (PAIR) {  // collective: both CTAs receive the same columns
      tmem_alloc_pair(tmem_slot, 2 * kAccCols);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(tmem_slot, 2 * kAccCols);
      tmem_relinquish();
    }
  }
  tc_fence_before();
  __syncthreads();
  uint32_t tmem;
  if constexpr (PAIR) {
    // barriers initialised and TMEM allocated in both CTAs before either signals the other; both
    // use the even CTA's TMEM address (the one its MMAs write)
    cg::this_cluster().sync();
    tc_fence_after();
    tmem = ld_dsmem_u32(dsmem_addr(tmem_slot, 0));
  } else {
    tc_fence_after();
    tmem = *tmem_slot;
  }

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
          if (prank == 0) mbar_arrive_expect_tx(&full[n_pre], PAIR ? 2 * stage_bytes : stage_bytes);
          for (int bx = 0; bx < a.kbox; ++bx) {
            const int kx = (pre_kb[n_pre] * a.kbox + bx) * kBK;
            if constexpr (PAIR)
              tma_load_2d_pair(st + bx * wbox_bytes, &map_w, dsmem_addr(&full[n_pre], 0), kx,
                               (2 * wt + prank) * kBM, pol_w);
            else
              tma_load_2d(st + bx * wbox_bytes, &map_w, &full[n_pre], kx, wt * a.nh * kBM, pol_w);
          }
        }
      }
      pdl_wait();
      for (int i = 0; i < n_pre; ++i) {
        const int tt_i = pre_tile[i] - (pre_tile[i] / a.n_ttiles) * a.n_ttiles;
        uint8_t* st = smem + i * stage_bytes;
        for (int bx = 0; bx < a.kbox; ++bx) {
          const int kx = (pre_kb[i] * a.kbox + bx) * kBK;
          if constexpr (PAIR)
            tma_load_2d_pair(st + a.kbox * wbox_bytes + bx * xbox_bytes, &map_x,
                             dsmem_addr(&full[i], 0), kx, tt_i * a.tt + prank * (a.tt / 2), pol_x);
          else
            tma_load_2d(st + a.kbox * wbox_bytes + bx * xbox_bytes, &map_x, &full[i], kx,
                        tt_i * a.tt, pol_x);
        }
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
          if (prank == 0) mbar_arrive_expect_tx(&full[s], PAIR ? 2 * stage_bytes : stage_bytes);
          for (int bx = 0; bx < a.kbox; ++bx) {
            const int ks = kb * a.kbox + bx;
            if constexpr (PAIR) {
              const uint32_t fb = dsmem_addr(&full[s], 0);
              tma_load_2d_pair(st + bx * wbox_bytes, &map_w, fb, ks * kBK, (2 * wt + prank) * kBM,
                               pol_w);
              tma_load_2d_pair(st + a.kbox * wbox_bytes + bx * xbox_bytes, &map_x, fb, ks * kBK,
                               tt_i * a.tt + prank * (a.tt / 2), pol_x);
            } else {
              tma_load_2d(st + bx * wbox_bytes, &map_w, &full[s], ks * kBK, wt * a.nh * kBM, pol_w);
              tma_load_2d(st + a.kbox * wbox_bytes + bx * xbox_bytes, &map_x, &full[s], ks * kBK,
                          tt_i * a.tt, pol_x);
            }
          }
          counts[0] = i + 1;
        }
      }
    }
  } else if (warp == 1) {
    pdl_wait();
    if (lane == 0) stamp_start(a.stamp);
    if (lane == 0 && prank == 0) {
      // ---- MMA issuer (PAIR: the even CTA, for both) ----
      const uint32_t idesc = idesc_bf16_f32(PAIR ? 2 * kBM : kBM, a.tt);
      const int ksub = a.kbox * (kBK / 16);
      int i = 0;
      bool ok = true;
      for (int j = 0; j < plan.count && ok; ++j) {
        int u, seg_end;
        seg_get(plan, j, u, seg_end);
        const int b = j % a.nbuf;
        if (!mbar_wait(&acce[b], ((j / a.nbuf) & 1) ^ 1, flags, a.budget)) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t d = tmem + b * a.accs;
        for (int uu = u; uu < seg_end; ++uu, ++i) {
          const int s = i % a.stages;
          const uint32_t ph = (i / a.stages) & 1;
          if (!mbar_wait(&full[s], ph, flags, a.budget)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sw = smem_u32(smem + s * stage_bytes);
          const uint32_t sx = sw + a.kbox * wbox_bytes;
          for (int kk = 0; kk < ksub; ++kk) {
            const uint32_t off = (kk & 3) * 32;
            const uint64_t bdesc = sdesc_k128(sx + (kk >> 2) * xbox_bytes + off);
            const uint32_t accum = (uu != u || kk != 0) ? 1u : 0u;
            if constexpr (PAIR) {
              mma_bf16_pair(d, sdesc_k128(sw + (kk >> 2) * wbox_bytes + off), bdesc, idesc, accum);
            } else {
              for (int h = 0; h < a.nh; ++h)
                mma_bf16(d + h * a.hoff,
                         sdesc_k128(sw + (kk >> 2) * wbox_bytes + h * kHalfW + off), bdesc, idesc,
                         accum);
            }
          }
          if constexpr (PAIR) mma_commit_pair(&empty[s], 3);  // both CTAs' stage s is free
          else mma_commit(&empty[s]);
          counts[1] = i + 1;
        }
        if (!ok) break;
        if constexpr (PAIR) mma_commit_pair(&accf[b], 3);
        else mma_commit(&accf[b]);
      }
      if (!ok) {
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
      }
      // arrives once every MMA issued above has completed
      if constexpr (PAIR) mma_commit_pair(done, 1);
      else mma_commit(done);
      volatile int no_abort = 0;
      if (!mbar_wait(done, 0, &no_abort, a.budget)) set_status(a.status, SPD_ETIMEOUT);
    }
  } else {
    pdl_wait();
    // ---- epilogue (warps 2..9; warp w reads TMEM lane quarter w % 4 and the 8-column groups of
    // parity (w - 2) / 4) ----
    const int q = warp & 3;
    const int half = (warp - 2) >> 2;
    const int row = q * 32 + lane;
    // Rotary table: where the CTA's only segment is a whole tile of a staged rotary epilogue, the
    // second TMEM accumulator is unused, and the epilogue warps, idle during the main loop, fill it
    // with the (cos, sin) of every 8-token group of their lanes (8 fp32 columns a group: the four
    // tokens' angles the lane evaluates in rope8). The epilogue then loads them beside the
    // accumulator instead of evaluating them after it is ready (the same function of the same
    // inputs: identical values).
    bool rtab = false;
    const uint32_t ttab = tmem + a.accs + (static_cast<uint32_t>(q * 32) << 16);
    if constexpr (EPI == EPI_QKV_BF16 || EPI == EPI_ROPE_BF16) {
      if (a.staged && plan.count == 1 && a.nbuf == 2 && a.nh == 1) {
        int u0s, u1s;
        seg_get(plan, 0, u0s, u1s);
        const int tile = u0s / a.n_kb;
        if (u0s == tile * a.n_kb && u1s - u0s == a.n_kb) {
          const int wt = tile / a.n_ttiles, tt_i = tile - wt * a.n_ttiles;
          const int tok0 = tt_i * a.tt, valid = min(a.tt, a.n_tok - tok0);
          const int n = (PAIR ? 2 * wt + prank : wt) * kBM + row;
          const bool second = EPI == EPI_QKV_BF16 && n >= a.split;
          const int nn = second ? n - a.split : n;
          if ((EPI == EPI_QKV_BF16 && !second) || nn < a.rope_rows) {  // warp-uniform
            rtab = true;
#pragma unroll 1
            for (int cc = half * 8; cc < valid; cc += 16) {
              float cm[4], sm[4];
              rope_angles4(a, nn, lane, tok0 + cc, [&](int t) { return a.pos ? a.pos[t] : 0; }, cm, sm);
              const float w[8] = {cm[0], sm[0], cm[1], sm[1], cm[2], sm[2], cm[3], sm[3]};
              tmem_st8(ttab + cc, w);
            }
            tmem_st_wait();
          }
        }
      }
    }
    for (int j = 0; j < plan.count; ++j) {
      int u, seg_end;
      seg_get(plan, j, u, seg_end);
      const int tile = u / a.n_kb;
      const int kb_lo = u - tile * a.n_kb;
      const int seg_len = seg_end - u;
      const int b = j % a.nbuf;
      const bool got = mbar_wait(&accf[b], (j / a.nbuf) & 1, flags, a.budget);
      if (epi_any(!got)) {  // every epilogue thread leaves together
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
        break;
      }
      tc_fence_after();
      if (a.cluster) break;  // cluster split-K: the accumulator is pushed after the role loops
      const int wt = tile / a.n_ttiles, tt_i = tile - wt * a.n_ttiles;
      const int tok0 = tt_i * a.tt;
      const int valid = min(a.tt, a.n_tok - tok0);
      const uint32_t tq = tmem + b * a.accs + (static_cast<uint32_t>(q * 32) << 16);
      const int blk0 = PAIR ? 2 * wt + prank : a.nh * wt;  // first 128-row block of this CTA
      // token metadata of this tile, staged once per segment
      const int et = threadIdx.x - 64;
      if (et < valid) {
        trow[et] = a.rows ? a.rows[tok0 + et] : tok0 + et;
        tpos[et] = a.pos ? a.pos[tok0 + et] : 0;
      }
      epi_bar();
      constexpr bool kStaged = EPI == EPI_QKV_BF16 || EPI == EPI_ROPE_BF16;
      if (kStaged && a.staged && j == plan.count - 1 && kb_lo == 0 && seg_len == a.n_kb) {
        // the CTA's last segment, whole: every MMA has completed, so the stage ring is idle and
        // holds the output block (bf16 rows of 256 bytes per 128 weight rows), which bulk copies
        // move out row by row instead of 2-byte scattered stores
        uint8_t* stg = smem;
        for (int h = 0; h < a.nh; ++h) {
          uint8_t* sh = stg + size_t(h) * a.tt * kStgPitch;
#pragma unroll 1
          for (int cc = half * 8; cc < valid; cc += 16) {
            float v[8];
            if (rtab) {  // j == 0, h == 0: the table of this segment
              float cs[8];
              tmem_ld8x2(tq + cc, v, ttab + cc, cs);
              stage8<EPI>(a, (blk0 + h) * kBM + row, lane, tok0 + cc, v, tpos, tok0, sh, cs);
            } else {
              tmem_ld8(tq + h * a.hoff + cc, v);
              stage8<EPI>(a, (blk0 + h) * kBM + row, lane, tok0 + cc, v, tpos, tok0, sh);
            }
          }
        }
        fence_proxy_async_smem();
        epi_bar();
        for (int h = 0; h < a.nh; ++h)
          stage_copy_out<EPI>(a, (blk0 + h) * kBM, et, tok0, valid, trow,
                              stg + size_t(h) * a.tt * kStgPitch);
      } else if ((kb_lo == 0 && seg_len == a.n_kb) || (EPI == EPI_ADD_F32 && !DET)) {
        for (int h = 0; h < a.nh; ++h) {
#pragma unroll 1
          for (int cc = half * 8; cc < valid; cc += 16) {
            float v[8];
            tmem_ld8(tq + h * a.hoff + cc, v);
            epilogue8<EPI>(a, (blk0 + h) * kBM + row, q, lane, blk0 + h, tok0 + cc, v, trow, tpos,
                           tok0);
          }
        }
      } else if (EPI != EPI_ADD_F32 && a.dpr) {
        // a remainder tile (dpr schedule): every contributor adds its partial into the tile's fp32
        // buffer at L2 ([tt tokens][CTA rows], token-major like the residual stream) with 16-byte
        // reductions after quad transposes; the last to arrive reads the sum, runs the epilogue
        // and leaves the buffer zero again. The order of the additions is not fixed (fp32 rounding
        // may differ in the last bits between runs).
        const int ctr = PAIR ? 2 * tile + prank : tile;
        const int ar = a.nh * kBM;  // floats per token row of the buffer
        float* acc = a.acc + size_t(ctr) * ar * a.tt;
        for (int h = 0; h < a.nh; ++h) {
#pragma unroll 1
          for (int cc = half * 8; cc < valid; cc += 16) {
            float v[8], w[8];
            tmem_ld8(tq + h * a.hoff + cc, v);
            quad_transpose8(v, w, lane);
            const int k = lane & 3, c0 = h * kBM + (row & ~3);
            red_add_v4(acc + size_t(cc + k) * ar + c0, w[0], w[1], w[2], w[3]);
            red_add_v4(acc + size_t(cc + 4 + k) * ar + c0, w[4], w[5], w[6], w[7]);
          }
        }
        __threadfence();  // the reductions are performed before the arrival below is seen
        epi_bar();
        if (threadIdx.x == 64) {
          const int old = atomicAdd(&a.counters[ctr], seg_len);
          flags[1] = (old + seg_len == a.n_kb);
        }
        epi_bar();
        if (flags[1]) {
          __threadfence();
          for (int h = 0; h < a.nh; ++h) {
            // the next group's sums are loaded before this group's epilogue (one L2 round trip
            // per group instead of two dependent ones)
            constexpr bool kPre = EPI == EPI_SWIGLU_BF16;  // the remainder schedule's GEMM
            float nx[8];
            if (kPre && half * 8 < valid) {
              const float* p0 = acc + size_t(half * 8) * ar + h * kBM + row;
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) nx[jj] = __ldcg(p0 + size_t(jj) * ar);
            }
#pragma unroll 1
            for (int cc = half * 8; cc < valid; cc += 16) {
              float* p = acc + size_t(cc) * ar + h * kBM + row;
              float v[8];
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) v[jj] = kPre ? nx[jj] : __ldcg(p + size_t(jj) * ar);
              if (kPre && cc + 16 < valid) {
                const float* pn = p + size_t(16) * ar;
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) nx[jj] = __ldcg(pn + size_t(jj) * ar);
              }
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) __stcg(p + size_t(jj) * ar, 0.0f);
              epilogue8<EPI>(a, (blk0 + h) * kBM + row, q, lane, blk0 + h, tok0 + cc, v, trow, tpos,
                             tok0);
            }
          }
          if (threadIdx.x == 64) a.counters[ctr] = 0;  // ready for the next launch
        }
      } else {
        // deterministic split tile: partial into this CTA's head (0) or tail (1) slot, laid out
        // [row half][4-column group][128 rows] of float4 (512 contiguous bytes per warp
        // instruction); the last arriver sums the partials in CTA order
        const size_t half_len = size_t(a.tt / 4) * kBM;
        const size_t slot_len = a.nh * half_len;
        float4* part = reinterpret_cast<float4*>(a.partial);
        float4* mine = part + size_t(2 * c + (tile == u0 / a.n_kb ? 0 : 1)) * slot_len;
        for (int h = 0; h < a.nh; ++h) {
#pragma unroll 1
          for (int cc = half * 8; cc < valid; cc += 16) {
            float v[8];
            tmem_ld8(tq + h * a.hoff + cc, v);
            float4* dst = mine + h * half_len + size_t(cc / 4) * kBM + row;
            __stcg(dst, make_float4(v[0], v[1], v[2], v[3]));
            __stcg(dst + kBM, make_float4(v[4], v[5], v[6], v[7]));
          }
        }
        __threadfence();
        epi_bar();
        const int ctr = PAIR ? 2 * tile + prank : tile;  // PAIR: each CTA's rows fix up alone
        if (threadIdx.x == 64) {
          const int old = atomicAdd(&a.counters[ctr], seg_len);
          flags[1] = (old + seg_len == a.n_kb);
        }
        epi_bar();
        if (flags[1]) {
          __threadfence();
          // contributors are work items c_first..c_last (this one: wc); the partial of item o
          // sits in the head or tail slot of its CTA (PAIR: the CTA holding these rows)
          const int c_first = cta_of_unit(tile * a.n_kb, a);
          const int c_last = cta_of_unit((tile + 1) * a.n_kb - 1, a);
          auto slot_of = [&](int o) {
            return 2 * (PAIR ? 2 * o + prank : o) + (tile == unit_lo(o, a) / a.n_kb ? 0 : 1);
          };
          if (c_last - c_first == 1) {
            // one other contributor (the usual case): its partial for eight 8-column groups in
            // flight at a time; a + b is exact in either order, so this matches the loop below
            const int o = (wc == c_first) ? c_last : c_first;
            const int os = slot_of(o);
            for (int h = 0; h < a.nh; ++h) {
              const float4* src = part + size_t(os) * slot_len + h * half_len + row;
#pragma unroll 1
              for (int cc0 = half * 8; cc0 < valid; cc0 += 128) {
                float4 x[16];
#pragma unroll
                for (int g = 0; g < 8; ++g) {
                  const int cc = cc0 + 16 * g;
                  if (cc < valid) {
                    x[2 * g] = __ldcg(src + size_t(cc / 4) * kBM);
                    x[2 * g + 1] = __ldcg(src + size_t(cc / 4 + 1) * kBM);
                  }
                }
#pragma unroll 1
                for (int g = 0; g < 8; ++g) {
                  const int cc = cc0 + 16 * g;
                  if (cc < valid) {
                    float v[8];
                    tmem_ld8(tq + h * a.hoff + cc, v);
                    add4(v, 0, x[0]);
                    add4(v, 4, x[1]);
                    epilogue8<EPI>(a, (blk0 + h) * kBM + row, q, lane, blk0 + h,
                                   tok0 + cc, v, trow, tpos, tok0);
                  }
                  // next group's data into the fixed slots (static register indices)
#pragma unroll
                  for (int k = 0; k < 14; ++k) x[k] = x[k + 2];
                }
              }
            }
          } else if (c_last - c_first == 2) {
            // two other contributors: two groups in flight, summed in CTA order
            // ((first + second) + third, this CTA's own partial in its place), as below
            const int own = wc - c_first;
            const int oa = (own == 0) ? c_first + 1 : c_first;  // first other contributor
            const int ob = (own == 2) ? c_first + 1 : c_last;   // second
            const int sa = slot_of(oa);
            const int sb = slot_of(ob);
            for (int h = 0; h < a.nh; ++h) {
              const float4* pa = part + size_t(sa) * slot_len + h * half_len + row;
              const float4* pb = part + size_t(sb) * slot_len + h * half_len + row;
#pragma unroll 1
              for (int cc0 = half * 8; cc0 < valid; cc0 += 32) {
                float4 xa[4], xb[4];
#pragma unroll
                for (int g = 0; g < 2; ++g) {
                  const int cc = cc0 + 16 * g;
                  if (cc < valid) {
                    xa[2 * g] = __ldcg(pa + size_t(cc / 4) * kBM);
                    xa[2 * g + 1] = __ldcg(pa + size_t(cc / 4 + 1) * kBM);
                    xb[2 * g] = __ldcg(pb + size_t(cc / 4) * kBM);
                    xb[2 * g + 1] = __ldcg(pb + size_t(cc / 4 + 1) * kBM);
                  }
                }
#pragma unroll 1
                for (int g = 0; g < 2; ++g) {
                  const int cc = cc0 + 16 * g;
                  if (cc < valid) {
                    float v[8];
                    tmem_ld8(tq + h * a.hoff + cc, v);
                    const float x1[8] = {xa[0].x, xa[0].y, xa[0].z, xa[0].w,
                                         xa[1].x, xa[1].y, xa[1].z, xa[1].w};
                    const float x2[8] = {xb[0].x, xb[0].y, xb[0].z, xb[0].w,
                                         xb[1].x, xb[1].y, xb[1].z, xb[1].w};
                    float acc[8];
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                      if (own == 0) acc[k] = (v[k] + x1[k]) + x2[k];
                      else if (own == 1) acc[k] = (x1[k] + v[k]) + x2[k];
                      else acc[k] = (x1[k] + x2[k]) + v[k];
                    }
                    epilogue8<EPI>(a, (blk0 + h) * kBM + row, q, lane, blk0 + h,
                                   tok0 + cc, acc, trow, tpos, tok0);
                  }
                  xa[0] = xa[2];
                  xa[1] = xa[3];
                  xb[0] = xb[2];
                  xb[1] = xb[3];
                }
              }
            }
          } else {
          for (int h = 0; h < a.nh; ++h) {
#pragma unroll 1
            for (int cc = half * 8; cc < valid; cc += 16) {
              float v[8], acc[8];
              tmem_ld8(tq + h * a.hoff + cc, v);
#pragma unroll
              for (int jj = 0; jj < 8; ++jj) acc[jj] = 0.0f;
              // contributors in CTA order, two partial tiles in flight at a time
#pragma unroll 1
              for (int o = c_first; o <= c_last; o += 2) {
                float4 x[4];
                const bool l0 = (o != wc), l1 = (o + 1 <= c_last) && (o + 1 != wc);
                if (l0) {
                  const int os = slot_of(o);
                  const float4* src =
                      part + size_t(os) * slot_len + h * half_len + size_t(cc / 4) * kBM + row;
                  x[0] = __ldcg(src);
                  x[1] = __ldcg(src + kBM);
                }
                if (l1) {
                  const int os = slot_of(o + 1);
                  const float4* src =
                      part + size_t(os) * slot_len + h * half_len + size_t(cc / 4) * kBM + row;
                  x[2] = __ldcg(src);
                  x[3] = __ldcg(src + kBM);
                }
                if (l0) {
                  add4(acc, 0, x[0]);
                  add4(acc, 4, x[1]);
                } else {
#pragma unroll
                  for (int jj = 0; jj < 8; ++jj) acc[jj] += v[jj];
                }
                if (o + 1 <= c_last) {
                  if (l1) {
                    add4(acc, 0, x[2]);
                    add4(acc, 4, x[3]);
                  } else {
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj) acc[jj] += v[jj];
                  }
                }
              }
              epilogue8<EPI>(a, (blk0 + h) * kBM + row, q, lane, blk0 + h, tok0 + cc,
                             acc, trow, tpos, tok0);
            }
          }
          }
          if (threadIdx.x == 64) a.counters[ctr] = 0;  // ready for the next launch
        }
      }
      tc_fence_before();
      epi_bar();  // trow / tpos / flags[1] are reused by the next segment
      if constexpr (PAIR) {  // one arrive per CTA on the even CTA's barrier
        if (threadIdx.x == 64) {
          if (prank == 0) mbar_arrive(&acce[b]);
          else mbar_arrive_cluster(dsmem_addr(&acce[b], 0));
        }
      } else {
        mbar_arrive(&acce[b]);
      }
    }
  }
  __syncthreads();
  if (!PAIR && a.cluster) {
    // cluster reduction, one 128-row half at a time; every thread of every CTA of the cluster
    // takes part in every barrier. Receive layout in each owner's ring: [sender][owned chunk][128
    // rows][kRecvPitch] fp32 (32 columns + 4 of padding: conflict-free 16-byte accesses).
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
    const bool epi = warp >= 2 && !flags[0];
    const int q = warp & 3, half = (warp - 2) >> 2, row = q * 32 + lane;
    for (int h = 0; h < a.nh; ++h) {
      cl.sync();  // every ring of the cluster is idle (h = 0) / its previous half consumed (h = 1)
      if (epi) {
        tc_fence_after();
        const uint32_t tq = tmem + h * a.hoff + (static_cast<uint32_t>(q * 32) << 16);
#pragma unroll 1
        for (int ci = half; ci * 32 < valid; ci += 2) {
          float v[32];
          tmem_ld32(tq + ci * 32, v);
          const int owner = ci % C, lc = ci / C;
          const uint32_t dst = dsmem_addr(
              recv + (size_t(r * cpo + lc) * kBM + row) * kRecvPitch, uint32_t(owner));
#pragma unroll
          for (int g = 0; g < 8; ++g)
            st_dsmem_v4(dst + g * 16,
                        make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]));
        }
      }
      cl.sync();  // all pushes of this half have landed
      if (epi) {
        const int n = (a.nh * wt + h) * kBM + row;
        // owned chunk lc covers columns (r + lc C) 32 .. +31; 8-column groups alternate between
        // the two warps of a lane quarter
#pragma unroll 1
        for (int gi = half; gi < 4 * cpo; gi += 2) {
          const int lc = gi >> 2, g8 = (gi & 3) * 8;
          const int col = (r + lc * C) * 32 + g8;
          if (col >= valid) continue;
          float acc[8];
#pragma unroll
          for (int jj = 0; jj < 8; ++jj) acc[jj] = 0.0f;
#pragma unroll 1
          for (int sdr = 0; sdr < C; ++sdr) {
            const float4* src = reinterpret_cast<const float4*>(
                recv + (size_t(sdr * cpo + lc) * kBM + row) * kRecvPitch + g8);
            add4(acc, 0, src[0]);
            add4(acc, 4, src[1]);
          }
          epilogue8<EPI>(a, n, q, lane, a.nh * wt + h, tok0 + col, acc, trow, tpos, tok0);
        }
      }
    }
  }
  if (threadIdx.x == 0 && flags[0] && prank == 0) {
    // drain: TMA loads issued but never consumed must land before the CTA exits (PAIR: the even
    // CTA's stage barriers count both CTAs' loads)
    for (int i = counts[1]; i < counts[0]; ++i) {
      volatile int no_abort = 0;
      mbar_wait(&full[i % a.stages], (i / a.stages) & 1, &no_abort, a.budget);
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x == 0) stamp_end(a.stamp);
  if constexpr (PAIR) {
    // the even CTA's MMAs have completed (its MMA thread waited above) and both CTAs' epilogues
    // are done before either CTA frees its TMEM or leaves (its shared memory feeds the MMAs)
    cg::this_cluster().sync();
    tc_fence_after();
    if (warp == 0) tmem_dealloc_pair(*tmem_slot, 2 * kAccCols);
  } else {
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem, 2 * kAccCols);
  }
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

int gemm_scratch_clear(const GemmScratch& s, cudaStream_t stream) {
  SPD_CUDA_TRY(cudaMemsetAsync(s.counters, 0, s.n_counters * sizeof(int), stream));
  if (s.acc_floats) SPD_CUDA_TRY(cudaMemsetAsync(s.acc, 0, s.acc_floats * sizeof(float), stream));
  return SPD_OK;
}

namespace {
std::atomic<int> g_deterministic{0};
}
int deterministic() { return g_deterministic.load(std::memory_order_relaxed); }
void set_deterministic(int on) { g_deterministic.store(on ? 1 : 0, std::memory_order_relaxed); }

size_t gemm_scratch_bytes() {
  return (kGemmSlotFloats + kGemmAccFloats) * sizeof(float) + kCounters * sizeof(int) + 768;
}

int make_weight_map(CUtensorMap* map, const void* w, int n_out, int k) {
  return make_map(map, w, k, n_out, kBM);
}

int make_operand_map(CUtensorMap* map, const void* ptr, int inner, int outer, int box_outer) {
  return make_map(map, ptr, inner, outer, box_outer);
}

namespace {

// ---- matrix-vector path (at most kGemvTok tokens, e.g. a decode step) ----------------------------
// With a handful of tokens the contraction is a pure weight stream: no tensor-core tile can be
// filled, and the tiled kernel's fixed costs (TMEM, barriers, a ring sized for wide tiles) and its
// shared-memory traffic per weight byte cap it well below the HBM roof. Here each CTA owns 32
// weight rows (warp w: rows 4w .. 4w + 3) over a range of K; every lane streams 16-byte chunks
// (eight bf16) so that one warp load covers 512 contiguous bytes of a row, with eight loads in
// flight per lane, and multiplies them with the tokens' chunks staged in shared memory (fp32
// accumulation, fixed order). The first batch of weight loads is issued before the grid waits
// on its predecessor (weights do not depend on it). The 32 row sums are then laid out as the
// tcgen05 accumulator would hold them (lane = row within the 32-row group, eight token columns)
// and go through the same fused epilogues. Residual (ADD) epilogues may split K over several CTAs
// (red.add, as in the tiled kernel); the others own whole rows.
constexpr int kGemvTok = 4;
constexpr int kGemvThreads = 256;
constexpr int kGemvChunk = 256;  // K elements per chunk column (32 lanes x 8 bf16)

__device__ __forceinline__ int4 ld_weights(const int4* p) {
  int4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.s32 {%0, %1, %2, %3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}
// acc + the dot product of eight bf16 pairs (w, x), element 2i in the low half of word i
__device__ __forceinline__ float dot8_bf16(const int4& w, const int4& x, float acc) {
  const uint32_t wu[4] = {uint32_t(w.x), uint32_t(w.y), uint32_t(w.z), uint32_t(w.w)};
  const uint32_t xu[4] = {uint32_t(x.x), uint32_t(x.y), uint32_t(x.z), uint32_t(x.w)};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    acc = fmaf(__uint_as_float(wu[i] << 16), __uint_as_float(xu[i] << 16), acc);
    acc = fmaf(__uint_as_float(wu[i] & 0xffff0000u), __uint_as_float(xu[i] & 0xffff0000u), acc);
  }
  return acc;
}

// NT: tokens computed (>= n_tok); CPR: chunks of a row per batch. A warp's work is a sequence of
// batches (row pair, block of CPR chunk columns). One register buffer per warp: latency is hidden
// by the number of resident warps (measured faster than double-buffering registers, which lowers
// occupancy).
template <int EPI, int NT, int CPR>
__global__ void __launch_bounds__(kGemvThreads)
    gemv_kernel(const uint16_t* __restrict__ w, const uint16_t* x, const KArgs a,
                int ksplit) {
  extern __shared__ __align__(16) uint8_t gsm[];
  __shared__ float red[32][NT];
  __shared__ int trow[kGemvTok], tpos[kGemvTok];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = blockIdx.x / ksplit, ks = blockIdx.x - grp * ksplit;
  const int n0 = grp * 32;
  const int C = a.k / kGemvChunk;
  const int kc0 = ks * C / ksplit, kc1 = (ks + 1) * C / ksplit, nc = kc1 - kc0;
  const int nblk = (nc + CPR - 1) / CPR;  // chunk blocks per row pair
  const int nb = 2 * nblk;                // batches of this warp (two row pairs)
  const int4* xs = reinterpret_cast<const int4*>(gsm);  // [NT][nc * 32] chunks of this K range
  const size_t wrow = size_t(a.k) / 8;                  // int4 per weight row
  const int4* wbase = reinterpret_cast<const int4*>(w) + size_t(kc0) * 32 + lane;
  // batch b: rows n0 + 4 warp + 2 (b / nblk) + {0, 1}, chunk columns (b % nblk) CPR + u
  auto load = [&](int4 (&buf)[2][CPR], int b) {
    const int rp = b / nblk, c0 = (b - rp * nblk) * CPR;
    const int r = n0 + 4 * warp + 2 * rp;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
      for (int u = 0; u < CPR; ++u)
        buf[h][u] = (c0 + u < nc && r + h < a.n_out)
                        ? ld_weights(wbase + size_t(r + h) * wrow + 32 * (c0 + u))
                        : make_int4(0, 0, 0, 0);
  };
  float acc[2][NT];
  auto compute = [&](const int4 (&buf)[2][CPR], int b) {
    const int rp = b / nblk, blk = b - rp * nblk, c0 = blk * CPR;
    if (blk == 0) {
#pragma unroll
      for (int t = 0; t < NT; ++t) acc[0][t] = acc[1][t] = 0.0f;
    }
#pragma unroll
    for (int u = 0; u < CPR; ++u) {
      const int c = c0 + u;
      if (c < nc) {
#pragma unroll
        for (int t = 0; t < NT; ++t) {
          const int4 xv = xs[t * nc * 32 + c * 32 + lane];
          acc[0][t] = dot8_bf16(buf[0][u], xv, acc[0][t]);
          acc[1][t] = dot8_bf16(buf[1][u], xv, acc[1][t]);
        }
      }
    }
    if (blk == nblk - 1) {  // the row pair is complete
#pragma unroll
      for (int t = 0; t < NT; ++t) {
        const float s0 = warp_sum_f(acc[0][t]), s1 = warp_sum_f(acc[1][t]);
        if (lane == 0) {
          red[4 * warp + 2 * rp][t] = s0;
          red[4 * warp + 2 * rp + 1][t] = s1;
        }
      }
    }
  };
  pdl_launch_dependents();
  int4 b0[2][CPR];
  load(b0, 0);  // weights do not depend on the predecessor: in flight before the wait
  pdl_wait();
  if (threadIdx.x == 0) stamp_start(a.stamp);
  if (a.norm_h) {  // the input RMSNorm of each token's fp32 row, computed by every CTA
    __shared__ float nred[kGemvThreads / 32][NT];
    __shared__ float ninv[NT];
#pragma unroll
    for (int t = 0; t < NT; ++t) {
      float ss = 0.0f;
      const int hrow = t < a.n_tok ? (a.norm_rows ? a.norm_rows[t] : t) : -1;  // -1: list padding
      if (hrow >= 0) {
        const float4* hr = reinterpret_cast<const float4*>(a.norm_h + size_t(hrow) * a.k);
        for (int c = threadIdx.x; c < a.k / 4; c += kGemvThreads) {
          const float4 v = hr[c];
          ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
      }
      ss = warp_sum_f(ss);
      if (lane == 0) nred[warp][t] = ss;
    }
    __syncthreads();
    if (threadIdx.x < NT) {
      float tot = 0.0f;
      for (int i = 0; i < kGemvThreads / 32; ++i) tot += nred[i][threadIdx.x];
      ninv[threadIdx.x] = rsqrtf(tot / float(a.k) + a.norm_eps);
    }
    __syncthreads();
    int4* xd = reinterpret_cast<int4*>(gsm);
    for (int e = threadIdx.x; e < NT * nc * 32; e += kGemvThreads) {
      const int t = e / (nc * 32), c = e - t * (nc * 32);
      int4 r = make_int4(0, 0, 0, 0);
      const int hrow = t < a.n_tok ? (a.norm_rows ? a.norm_rows[t] : t) : -1;
      if (hrow >= 0) {
        const size_t k0 = size_t(kc0 * 32 + c) * 8;
        const float* hr = a.norm_h + size_t(hrow) * a.k + k0;
        const float4 v0 = reinterpret_cast<const float4*>(hr)[0], v1 = reinterpret_cast<const float4*>(hr)[1];
        const uint4 gg = *reinterpret_cast<const uint4*>(a.norm_gain + k0);
        const float inv = ninv[t];
        const float hv[8] = {v0.x, v0.y, v0.z, v0.w, v1.x, v1.y, v1.z, v1.w};
        const uint32_t gw[4] = {gg.x, gg.y, gg.z, gg.w};
        uint32_t pk[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {  // the same products and rounding as the RMSNorm kernel
          const __nv_bfloat162 b2 = __floats2bfloat162_rn(hv[2 * i] * inv * __uint_as_float(gw[i] << 16),
                                                          hv[2 * i + 1] * inv * __uint_as_float(gw[i] & 0xffff0000u));
          pk[i] = *reinterpret_cast<const uint32_t*>(&b2);
        }
        r = make_int4(int(pk[0]), int(pk[1]), int(pk[2]), int(pk[3]));
      }
      xd[e] = r;
    }
    if (threadIdx.x < a.n_tok) {
      trow[threadIdx.x] = a.rows ? a.rows[threadIdx.x] : threadIdx.x;
      tpos[threadIdx.x] = a.pos ? a.pos[threadIdx.x] : 0;
    }
  } else {  // tokens' chunks of this K range; token rows past n_tok are zeros
    int4* xd = reinterpret_cast<int4*>(gsm);
    for (int e = threadIdx.x; e < NT * nc * 32; e += kGemvThreads) {
      const int t = e / (nc * 32), c = e - t * (nc * 32);
      xd[e] = t < a.n_tok ? reinterpret_cast<const int4*>(x + size_t(t) * a.k)[kc0 * 32 + c]
                          : make_int4(0, 0, 0, 0);
    }
    if (threadIdx.x < a.n_tok) {
      trow[threadIdx.x] = a.rows ? a.rows[threadIdx.x] : threadIdx.x;
      tpos[threadIdx.x] = a.pos ? a.pos[threadIdx.x] : 0;
    }
  }
  __syncthreads();
#pragma unroll 1
  for (int b = 0; b < nb; ++b) {
    if (b > 0) load(b0, b);
    compute(b0, b);
  }
  __syncthreads();
  if (warp == 0) {
    float v[8];
#pragma unroll
    for (int t = 0; t < 8; ++t) v[t] = t < NT ? red[lane][t] : 0.0f;
    epilogue8<EPI>(a, n0 + lane, (n0 >> 5) & 3, lane, n0 >> 7, 0, v, trow, tpos, 0);
    if (lane == 0) stamp_end(a.stamp);
  }
}

using GemvFn = void (*)(const uint16_t*, const uint16_t*, KArgs, int);
template <int NT, int CPR>
GemvFn gemv_for(int epi) {
  switch (epi) {
    case EPI_F32: return gemv_kernel<EPI_F32, NT, CPR>;
    case EPI_ADD_F32: return gemv_kernel<EPI_ADD_F32, NT, CPR>;
    case EPI_SWIGLU_BF16: return gemv_kernel<EPI_SWIGLU_BF16, NT, CPR>;
    case EPI_QKV_BF16: return gemv_kernel<EPI_QKV_BF16, NT, CPR>;
    default: return nullptr;
  }
}

using KernelFn = void (*)(CUtensorMap, CUtensorMap, KArgs);

template <bool PAIR>
KernelFn kernel_for(int epi) {
  switch (epi) {
    case EPI_F32: return gemm_sk_kernel<EPI_F32, PAIR>;
    case EPI_BF16: return gemm_sk_kernel<EPI_BF16, PAIR>;
    case EPI_BIAS_BF16: return gemm_sk_kernel<EPI_BIAS_BF16, PAIR>;
    case EPI_BIAS_GELU_BF16: return gemm_sk_kernel<EPI_BIAS_GELU_BF16, PAIR>;
    case EPI_ADD_F32: return gemm_sk_kernel<EPI_ADD_F32, PAIR, false>;
    case EPI_ROPE_BF16: return gemm_sk_kernel<EPI_ROPE_BF16, PAIR>;
    case EPI_SWIGLU_BF16: return gemm_sk_kernel<EPI_SWIGLU_BF16, PAIR>;
    case EPI_QKV_BF16: return gemm_sk_kernel<EPI_QKV_BF16, PAIR>;
    case EPI_LSE_F32: return gemm_sk_kernel<EPI_LSE_F32, PAIR>;
    default: return nullptr;
  }
}
KernelFn kernel_for(int epi, bool pair, bool det = false) {
  if (det && epi == EPI_ADD_F32)
    return pair ? gemm_sk_kernel<EPI_ADD_F32, true, true> : gemm_sk_kernel<EPI_ADD_F32, false, true>;
  return pair ? kernel_for<true>(epi) : kernel_for<false>(epi);
}

// Sets the shared-memory limit of every instance once; returns the first error.
cudaError_t set_kernel_attributes() {
  static std::once_flag once;
  static cudaError_t err = cudaSuccess;
  std::call_once(once, [] {
    for (int e : {int(EPI_F32), int(EPI_BF16), int(EPI_BIAS_BF16), int(EPI_BIAS_GELU_BF16),
                  int(EPI_ADD_F32), int(EPI_ROPE_BF16), int(EPI_SWIGLU_BF16),
                  int(EPI_QKV_BF16), int(EPI_LSE_F32)}) {
      for (int v = 0; v < 4; ++v) {
        const bool pair = v & 1, det = v & 2;
        const cudaError_t r =
            cudaFuncSetAttribute(reinterpret_cast<const void*>(kernel_for(e, pair, det)),
                                 cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 kSmemPipe + 1024 + 256 + 16384);
        if (r != cudaSuccess && err == cudaSuccess) err = r;
      }
    }
  });
  return err;
}

// Clusters of C CTAs (at the largest shared-memory size) that the GPU holds at once. Not every
// GPC holds the same number of them, so 152 SMs need not hold 152 / C clusters.
int max_active_clusters(int C) {
  static int cache[9] = {0};
  static std::once_flag once;
  std::call_once(once, [] {
    for (int cs = 2; cs <= 8; cs *= 2) {
      cudaLaunchConfig_t cfg = {};
      cfg.gridDim = dim3(cs);
      cfg.blockDim = dim3(kThreads);
      cfg.dynamicSmemBytes = kSmemPipe + 1024 + 256 + 2048;
      cudaLaunchAttribute attr[1];
      attr[0].id = cudaLaunchAttributeClusterDimension;
      attr[0].val.clusterDim.x = cs;
      attr[0].val.clusterDim.y = 1;
      attr[0].val.clusterDim.z = 1;
      cfg.attrs = attr;
      cfg.numAttrs = 1;
      int n = 0;
      if (cudaOccupancyMaxActiveClusters(&n,
                                         reinterpret_cast<const void*>(kernel_for(EPI_F32, false)),
                                         &cfg) != cudaSuccess) {
        cudaGetLastError();
        n = 0;
      }
      cache[cs] = n;
    }
  });
  return cache[C];
}

}  // namespace

namespace {
// Algorithmic work of one GEMM call (valid output columns only; weights, activations and results
// move once; fused QKV: query rows count for the query tokens only).
void gemm_work(const GemmProblem& p, double* flops, double* bytes) {
  const double cols = (p.epi == EPI_SWIGLU_BF16) ? 2.0 * p.out_cols : double(p.n_out);
  const double out_cols = (p.epi == EPI_SWIGLU_BF16) ? double(p.out_cols) : double(p.n_out);
  const double ob = (p.epi == EPI_F32) ? 4.0 : (p.epi == EPI_ADD_F32) ? 8.0 : (p.epi == EPI_LSE_F32) ? 0.5 : 2.0;
  double tok_cols = double(p.n_tok) * cols, tok_out = double(p.n_tok) * out_cols;
  if (p.epi == EPI_QKV_BF16) {
    tok_cols = double(p.n_tok_out) * p.split + double(p.n_tok) * (p.n_out - p.split);
    tok_out = tok_cols;
  }
  *flops = 2.0 * tok_cols * p.k;
  *bytes = 2.0 * cols * p.k + 2.0 * p.n_tok * p.k + ob * tok_out;
}
void trace_gemm(int slot, const GemmProblem& p, cudaStream_t stream) {
  if (slot < 0) return;
  double fl, by;
  gemm_work(p, &fl, &by);
  trace_end(slot, stream, TR_GEMM, fl, by);
}
unsigned long long* gemm_stamp(const GemmProblem& p) {
  double fl, by;
  gemm_work(p, &fl, &by);
  return stamp_slot(TR_GEMM, fl, by);
}

// 16-byte residual reductions need 4-column groups that start 16-byte aligned in every row
bool vec_red_ok(const GemmProblem& p) {
  return p.epi == EPI_ADD_F32 && p.n_out % 4 == 0 && p.ldo % 4 == 0 &&
         (reinterpret_cast<uintptr_t>(p.out) & 15) == 0;
}

bool gemv_eligible(const GemmProblem& p) {
  if (p.norm_h && ((reinterpret_cast<uintptr_t>(p.norm_h) | reinterpret_cast<uintptr_t>(p.norm_gain)) & 15))
    return false;
  return p.n_tok <= kGemvTok && p.w && p.k % kGemvChunk == 0 &&
         (reinterpret_cast<uintptr_t>(p.w) & 15) == 0 && (reinterpret_cast<uintptr_t>(p.x) & 15) == 0 &&
         gemv_for<1, 4>(p.epi) != nullptr;
}

int gemv_run(const GemmProblem& p, const GemmScratch& s, cudaStream_t stream) {
  KArgs a{};
  a.n_out = p.n_out;
  a.n_tok = p.n_tok;
  a.k = p.k;
  a.out = p.out;
  a.ldo = p.ldo;
  a.out2 = p.out2;
  a.ldo2 = p.ldo2;
  a.split = p.split;
  a.rows = p.rows;
  a.rows2 = p.rows2;
  a.bias = p.bias;
  a.pos = p.pos;
  a.rope = reinterpret_cast<const float2*>(p.rope);
  a.rope_rows = p.rope_rows;
  a.head_dim = p.head_dim;
  a.out_cols = p.out_cols;
  a.status = s.status;
  a.norm_h = p.norm_h;
  a.norm_gain = p.norm_gain;
  a.norm_rows = p.norm_rows;
  a.norm_eps = p.norm_eps;
  a.stamp = gemm_stamp(p);
  a.vec_red = vec_red_ok(p);
  a.determ = deterministic();
  const int groups = (p.n_out + 31) / 32, C = p.k / kGemvChunk;
  // residual epilogues split K until about one CTA per SM streams (each at least one chunk column;
  // two per SM measured slower at the decoder's O and down shapes: shorter rows per CTA)
  int ksplit = 1;
  if (p.epi == EPI_ADD_F32 && !a.determ)
    while (groups * ksplit < num_sms() && ksplit * 2 <= C && ksplit < 8) ksplit *= 2;
  const bool one = p.n_tok == 1;
  const int nt = one ? 1 : kGemvTok;
  const size_t smem = size_t(nt) * ((C + ksplit - 1) / ksplit) * kGemvChunk * sizeof(uint16_t);
  const GemvFn kern = one ? gemv_for<1, 4>(p.epi) : gemv_for<kGemvTok, 4>(p.epi);
  static std::once_flag once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(once, [] {
    for (int e : {int(EPI_F32), int(EPI_ADD_F32), int(EPI_SWIGLU_BF16), int(EPI_QKV_BF16)})
      for (GemvFn f : {gemv_for<1, 4>(e), gemv_for<kGemvTok, 4>(e)}) {
        const cudaError_t r = cudaFuncSetAttribute(reinterpret_cast<const void*>(f),
                                                   cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                   200 * 1024);
        if (r != cudaSuccess && attr_err == cudaSuccess) attr_err = r;
      }
  });
  if (attr_err != cudaSuccess)
    return fail(SPD_ECUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(attr_err));
  if (smem > 200 * 1024) return fail(SPD_EUNSUPPORTED, "GEMV K range too long");
  const int slot = trace_begin(stream);
  SPD_CUDA_TRY(launch_pdl(kern, dim3(groups * ksplit), dim3(kGemvThreads), smem, stream,
                          static_cast<const uint16_t*>(p.w), static_cast<const uint16_t*>(p.x), a,
                          ksplit));
  trace_gemm(slot, p, stream);
  return SPD_OK;
}
}  // namespace

bool gemm_fuses_norm(const GemmProblem& p) { return p.n_tok > 0 && gemv_eligible(p); }

int gemm_run(const GemmProblem& p, const GemmScratch& s, cudaStream_t stream) {
  if (p.n_tok <= 0 || p.n_out <= 0) return SPD_OK;
  if (p.k <= 0) return fail(SPD_EINVAL, "GEMM K must be positive");
  if (!kernel_for(p.epi, false)) return fail(SPD_EINVAL, "unknown GEMM epilogue %d", p.epi);
  if (!p.map_w && !p.w) return fail(SPD_EINVAL, "GEMM without weights");
  if (gemv_eligible(p)) return gemv_run(p, s, stream);
  if (p.norm_h) return fail(SPD_EINVAL, "input RMSNorm fusion needs the matrix-vector path");
  if (cudaError_t e = set_kernel_attributes())
    return fail(SPD_ECUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(e));
  KArgs a{};
  a.n_out = p.n_out;
  a.n_tok = p.n_tok;
  a.k = p.k;
  a.n_ttiles = (p.n_tok + 255) / 256;
  a.tt = ((p.n_tok + a.n_ttiles - 1) / a.n_ttiles + 31) / 32 * 32;
  const int sms = num_sms();
  // CTA pairs (M = 256 over two SMs) for token tiles of at least 128, except where the tiles are
  // so few that only the cluster reduction of split-K partials fills the GPU (non-residual
  // epilogues): there the single-CTA kernel runs.
  const int slots = sms / 2;  // pairs the GPU holds at once
  const long long pair_tiles = (long long)((p.n_out + 2 * kBM - 1) / (2 * kBM)) * a.n_ttiles;
  // Deterministic mode: residual GEMMs that few also take the single-CTA kernel, whose cluster
  // reduction sums the split partials in rank order on every CTA of the cluster at once (the
  // ordered stream-K fixup of the pair kernel leaves each tile's sum to one CTA).
  const bool pair = a.tt >= 128 &&
                    !((p.epi != EPI_ADD_F32 || deterministic()) && pair_tiles * 2 <= slots);
  // 256-row tiles in one CTA for token tiles of at most 64: their stages are mostly weights, and
  // two MMAs per token box double the weight bytes per stage (needs the row-major pointer)
  a.nh = (!pair && a.tt <= 64 && p.w) ? 2 : 1;
  const int tile_rows = pair ? 2 * kBM : a.nh * kBM;  // weight rows per work item
  const int cta_rows = pair ? kBM : tile_rows;          // ... per CTA
  const int wbox = (pair ? 1 : a.nh) * kHalfW;
  const int xrows = pair ? a.tt / 2 : a.tt;            // token rows per CTA
  auto stages_for = [&](int kb) {
    return std::min(kMaxStages, kSmemPipe / (kb * (wbox + xrows * 128)));
  };
  // 128-wide k-blocks (256 contiguous bytes of every weight row per stage) when two stages fit
  a.kbox = (p.k > kBK && stages_for(2) >= 2) ? 2 : 1;
  a.n_kb = (p.k + a.kbox * kBK - 1) / (a.kbox * kBK);
  a.stages = stages_for(a.kbox);
  const int stage_bytes = a.kbox * (wbox + xrows * 128);
  // TMEM: 512 columns. Single CTA: two accumulator buffers of 256 unless a 256-row tile is wider
  // than 128 tokens; the second 128-row half sits 128 or 256 columns after the first. Pair: two
  // buffers of 256 (each CTA's TMEM holds its 128 rows).
  if (pair) {
    a.nbuf = 2;
    a.accs = kAccCols;
    a.hoff = 0;
  } else {
    a.nbuf = (a.nh * a.tt <= 256) ? 2 : 1;
    a.accs = kAccCols;
    a.hoff = a.tt <= 128 ? 128 : 256;
  }
  CUtensorMap map_w, map_x;
  if (cta_rows == kBM && p.map_w) {
    map_w = *p.map_w;
  } else if (int rc = make_map(&map_w, p.w, p.k, p.n_out, cta_rows)) {
    return rc;
  }
  if (int rc = make_map(&map_x, p.x, p.k, p.n_tok, xrows)) return rc;
  const int n_wtiles = (p.n_out + tile_rows - 1) / tile_rows;
  const long long tiles = (long long)n_wtiles * a.n_ttiles;
  if (tiles * (pair ? 2 : 1) > s.n_counters)
    return fail(SPD_EUNSUPPORTED, "GEMM has too many output tiles");
  const long long units = tiles * a.n_kb;
  if (units > 0x3fffffffLL) return fail(SPD_EUNSUPPORTED, "GEMM too large");
  a.units = int(units);
  const int work_slots = pair ? slots : sms;  // work items the GPU holds at once
  // split-K when the tiles fill at most half the work slots. ADD epilogues: the most work items
  // per tile (a power of two, at least two k-blocks each) that still fit. Others (single CTA):
  // the largest C in {2, 4, 8} with at least one k-block per CTA whose clusters all fit on the
  // GPU at once.
  a.csplit = 1;
  a.cluster = 0;
  a.determ = deterministic();
  if (tiles * 2 <= work_slots && p.epi == EPI_ADD_F32 && !a.determ) {
    int C = 2;
    while (tiles * C * 2 <= work_slots && C * 4 <= a.n_kb) C *= 2;
    if (C * 2 <= a.n_kb) a.csplit = C;
  } else if (!pair && tiles * 2 <= sms) {
    for (int C = 8; C >= 2; C /= 2) {
      // the ring receives C copies of each CTA's share of 32-column chunks ([128][36] fp32 each)
      const int chunks = a.tt / 32, cpo = (chunks + C - 1) / C;
      const size_t recv = size_t(C) * cpo * kBM * kRecvPitch * sizeof(float);
      if (C <= a.n_kb && tiles * C <= sms && tiles <= max_active_clusters(C) &&
          recv <= size_t(a.stages) * stage_bytes) {
        a.csplit = C;
        a.cluster = 1;
        break;
      }
    }
  }
  // stream-K: one work item per slot with at least 2 units each; every CTA owns two partial
  // slots (head, tail) of its rows x the token tile
  long long grid = work_slots;
  if (grid > (units + 1) / 2) grid = (units + 1) / 2;
  const size_t per_item = size_t(2) * a.tt * tile_rows;  // both slots of every CTA of the item
  if (size_t(grid) * per_item > s.partial_floats) grid = s.partial_floats / per_item;
  if (grid < 1) grid = 1;
  if (units * (grid + 1) >= (1LL << 31)) return fail(SPD_EUNSUPPORTED, "GEMM too large");
  // data-parallel + remainder (seg_plan_dpr) instead of stream-K for non-residual epilogues: W
  // whole tiles per work item, the R leftover tiles split in K over all items, their partial sums
  // accumulated at L2 (no fp32 partials stored per CTA and read back by one fixup CTA)
  a.dpr = 0;
  a.rem_tiles = 0;
  a.whole = 0;
  a.acc = s.acc;
  if (a.csplit == 1 && p.epi != EPI_ADD_F32 && tiles > work_slots && !a.determ) {
    const long long W = tiles / work_slots, R = tiles - W * work_slots;
    const size_t acc_need = size_t(R) * tile_rows * a.tt;
    // only a thin remainder (each item's share at most a quarter of a tile's k-blocks): with more,
    // stream-K's ordered fixups beat the L2 reductions (measured on the dense LLaVA step)
    if (R > 0 && R * 4 <= work_slots && R * a.n_kb >= 2 * work_slots && acc_need <= s.acc_floats) {
      a.dpr = 1;
      a.rem_tiles = int(R);
      a.whole = int(W);
      grid = work_slots;
    }
  }
  if (a.csplit > 1) {
    grid = tiles * a.csplit;
  } else if (a.dpr) {
    // grid set above
  } else if (tiles <= work_slots && tiles * 2 > work_slots && a.tt >= 128) {
    // between half and all of the work slots' worth of wide tiles: one whole tile per work item.
    // Stream-K's balance would split most tiles two or three ways, and the fixups of wide token
    // tiles cost more than the idle SMs do.
    grid = tiles;
  }
  a.grid = int(grid);
  const KernelFn kern = kernel_for(p.epi, pair, a.determ);
  a.out = p.out;
  a.ldo = p.ldo;
  a.out2 = p.out2;
  a.ldo2 = p.ldo2;
  a.split = p.split;
  a.rows = p.rows;
  a.rows2 = p.rows2;
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
  a.stamp = gemm_stamp(p);
  a.vec_red = vec_red_ok(p);
  {
    // staged rotary epilogues: whole 128-column output blocks of 16-byte aligned rows, the block
    // of every token of the tile fitting in the idle stage ring
    const bool rot = p.epi == EPI_QKV_BF16 || p.epi == EPI_ROPE_BF16;
    const bool al = ((reinterpret_cast<uintptr_t>(p.out) | reinterpret_cast<uintptr_t>(p.out2)) & 15) == 0 &&
                    p.ldo % 8 == 0 && (p.epi != EPI_QKV_BF16 || p.ldo2 % 8 == 0);
    a.staged = rot && al && !a.cluster && p.n_out % kBM == 0 && (p.epi != EPI_QKV_BF16 || p.split % kBM == 0) &&
               size_t(a.nh) * a.tt * kStgPitch <= size_t(a.stages) * stage_bytes;
  }

  const size_t smem = size_t(a.stages) * stage_bytes + 1024 + 256 + 2048;
  const int slot = trace_begin(stream);
  {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(pair ? 2 * a.grid : a.grid);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = pair ? 2 : (a.cluster ? a.csplit : 1);
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    SPD_CUDA_TRY(cudaLaunchKernelEx(&cfg, kern, map_w, map_x, a));
  }
  trace_gemm(slot, p, stream);
  return SPD_OK;
}

}  // namespace spd
