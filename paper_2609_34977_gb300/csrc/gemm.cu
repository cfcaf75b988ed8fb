// tcgen05 bf16 GEMM for the decoder's dense contractions: out = epilogue(X W^T).
//
// Prefill after pruning has few token rows (a few hundred) against large weight matrices, so the
// contraction is weight-stream bound. The kernel therefore puts the WEIGHTS on the MMA's M side
// (128 weight rows per CTA tile) and the tokens on the N side (up to 256 per tile): one CTA reads
// each weight tile from HBM exactly once and every token of the batch reuses it.
//
//   warp 0 lane 0 : TMA producer   - weight box 128 x 64 and token boxes 32 x 64 per stage
//   warp 1 lane 0 : MMA issuer     - 4 x tcgen05.mma (K = 16) per stage into a TMEM accumulator
//   warps 0..3    : epilogue       - tcgen05.ld of 32 lanes x 32 columns, fused epilogue, stores
//
// Split-K: when the tile count leaves SMs idle, K is split; every split stores its fp32 partial
// tile, and the last CTA to arrive on the tile's counter sums the partials in split order (a
// deterministic result) and runs the epilogue.
#include <cuda_bf16.h>
#include <math.h>
#include <stdio.h>

#include <mutex>

#include "internal.h"
#include "ptx.cuh"

namespace spd {
namespace {

constexpr int kBM = 128;            // weight rows per tile (MMA M)
constexpr int kBK = 64;             // K elements per stage (one 128-byte swizzle row)
constexpr int kWBytes = kBM * 128;  // weight box bytes per stage
constexpr int kXRows = 32;          // token rows per TMA box
constexpr int kXBoxBytes = kXRows * 128;
constexpr int kMaxStages = 8;
constexpr int kSmemPipe = 196608;   // bytes of the stage ring
constexpr int kTmemCols = 256;
constexpr size_t kPartialFloats = size_t(16) << 20;  // 64 MB of split-K partials
constexpr int kCounters = 1 << 16;

struct KArgs {
  int n_out, n_tok, k, tt, n_kb, splits, kbps, stages, epi, ldo, rope_rows, head_dim, out_cols,
      n_ttiles;
  void* out;
  const int32_t* rows;
  const uint16_t* bias;
  const int32_t* pos;
  const float* inv_freq;
  float* partial;
  int* counters;
  int* status;
  long long budget;
};

__device__ __forceinline__ float gelu_erf(float x) {
  return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}

// Applies the epilogue to 32 consecutive tokens t0..t0+31 of this thread's weight row n.
__device__ __forceinline__ void epilogue_chunk(const KArgs& a, int n, int warp, int lane,
                                               int w_tile, int t0, const float (&v)[32]) {
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
          const int r = a.rows ? a.rows[t] : t;
          float* p = o + size_t(r) * a.ldo + n;
          if (a.epi == EPI_ADD_F32) *p += v[j];
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
          const int r = a.rows ? a.rows[t] : t;
          float x = v[j] + b;
          if (a.epi == EPI_BIAS_GELU_BF16) x = gelu_erf(x);
          o[size_t(r) * a.ldo + n] = __float2bfloat16_rn(x);
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
        const float inv = a.inv_freq[jf];
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const float p = __shfl_xor_sync(0xffffffffu, v[j], 16);
          const int t = t0 + j;
          if (t < nt) {
            float s, c;
            sincosf(static_cast<float>(a.pos[t]) * inv, &s, &c);
            const float y = (lane < 16) ? v[j] * c - p * s : v[j] * c + p * s;
            const int r = a.rows ? a.rows[t] : t;
            o[size_t(r) * a.ldo + col] = __float2bfloat16_rn(y);
          }
        }
      } else {
#pragma unroll
        for (int j = 0; j < 32; ++j) {
          const int t = t0 + j;
          if (t < nt) {
            const int r = a.rows ? a.rows[t] : t;
            o[size_t(r) * a.ldo + n] = __float2bfloat16_rn(v[j]);
          }
        }
      }
      return;
    }
    case EPI_SWIGLU_BF16: {
      __nv_bfloat16* o = static_cast<__nv_bfloat16*>(a.out);
      const int f = w_tile * 64 + warp * 16 + (lane & 15);
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float u = __shfl_xor_sync(0xffffffffu, v[j], 16);
        const int t = t0 + j;
        if (lane < 16 && t < nt && f < a.out_cols) {
          const float g = v[j];
          const int r = a.rows ? a.rows[t] : t;
          o[size_t(r) * a.ldo + f] = __float2bfloat16_rn(g / (1.0f + expf(-g)) * u);
        }
      }
      return;
    }
    default:
      return;
  }
}

__global__ void __launch_bounds__(128, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap map_w,
                   const __grid_constant__ CUtensorMap map_x, const KArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~uintptr_t(1023));
  const uint32_t stage_bytes = kWBytes + a.tt * 128;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + a.stages * stage_bytes);
  uint64_t* empty = full + kMaxStages;
  uint64_t* accum = empty + kMaxStages;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(accum + 1);
  volatile int* flags = reinterpret_cast<volatile int*>(tmem_slot + 1);  // [0] abort [1] last

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int t_tile = blockIdx.x, w_tile = blockIdx.y, split = blockIdx.z;
  const int kb0 = split * a.kbps;
  const int nk = min(a.n_kb, kb0 + a.kbps) - kb0;
  const int tok0 = t_tile * a.tt;
  const int tok_valid = min(a.tt, a.n_tok - tok0);
  const int x_boxes = (tok_valid + kXRows - 1) / kXRows;
  const uint32_t tx_bytes = kWBytes + x_boxes * kXBoxBytes;

  if (threadIdx.x == 0) {
    for (int s = 0; s < a.stages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accum, 1);
    flags[0] = 0;
    flags[1] = 0;
    fence_mbar_init();
    prefetch_tmap(&map_w);
    prefetch_tmap(&map_x);
  }
  if (warp == 0) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0 && lane == 0) {
    // ---- TMA producer ----
    const uint64_t pol_w = policy_evict_first(), pol_x = policy_evict_last();
    for (int i = 0; i < nk; ++i) {
      const int s = i % a.stages;
      const uint32_t ph = (i / a.stages) & 1;
      if (!mbar_wait(&empty[s], ph ^ 1, flags, a.budget)) {
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
        break;
      }
      uint8_t* st = smem + s * stage_bytes;
      mbar_arrive_expect_tx(&full[s], tx_bytes);
      const int kx = (kb0 + i) * kBK;
      tma_load_2d(st, &map_w, &full[s], kx, w_tile * kBM, pol_w);
      for (int c = 0; c < x_boxes; ++c)
        tma_load_2d(st + kWBytes + c * kXBoxBytes, &map_x, &full[s], kx, tok0 + c * kXRows, pol_x);
    }
  } else if (warp == 1 && lane == 0) {
    // ---- MMA issuer ----
    const uint32_t idesc = idesc_bf16_f32(kBM, a.tt);
    for (int i = 0; i < nk; ++i) {
      const int s = i % a.stages;
      const uint32_t ph = (i / a.stages) & 1;
      if (!mbar_wait(&full[s], ph, flags, a.budget)) {
        flags[0] = 1;
        set_status(a.status, SPD_ETIMEOUT);
        break;
      }
      tc_fence_after();
      const uint32_t sa = smem_u32(smem + s * stage_bytes);
#pragma unroll
      for (int kk = 0; kk < kBK / 16; ++kk)
        mma_bf16(tmem, sdesc_k128(sa + kk * 32), sdesc_k128(sa + kWBytes + kk * 32), idesc,
                 (i | kk) != 0);
      mma_commit(&empty[s]);
    }
    mma_commit(accum);  // arrives once every MMA above has completed
  }
  __syncwarp();

  // ---- epilogue ----
  if (!mbar_wait(accum, 0, flags, a.budget)) {
    flags[0] = 1;
    set_status(a.status, SPD_ETIMEOUT);
  }
  tc_fence_after();
  __syncthreads();
  bool run = (flags[0] == 0);
  const int row = warp * 32 + lane;
  const int n = w_tile * kBM + row;
  const uint32_t tw = tmem + (static_cast<uint32_t>(warp * 32) << 16);
  const int tile_id = w_tile * a.n_ttiles + t_tile;
  if (run && a.splits > 1) {
    float* mine = a.partial + (size_t(tile_id) * a.splits + split) * size_t(a.tt) * kBM;
    for (int c = 0; c < tok_valid; c += 32) {
      float v[32];
      tmem_ld32(tw + c, v);
#pragma unroll
      for (int j = 0; j < 32; ++j) mine[size_t(c + j) * kBM + row] = v[j];
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      const int old = atomicAdd(&a.counters[tile_id], 1);
      flags[1] = (old == a.splits - 1);
    }
    __syncthreads();
    run = (flags[1] != 0);
    if (run) __threadfence();
  }
  if (run) {
    for (int c = 0; c < tok_valid; c += 32) {
      float v[32];
      tmem_ld32(tw + c, v);
      if (a.splits > 1) {
        float acc[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) acc[j] = 0.0f;
        for (int s = 0; s < a.splits; ++s) {
          if (s == split) {
#pragma unroll
            for (int j = 0; j < 32; ++j) acc[j] += v[j];
          } else {
            const float* p =
                a.partial + ((size_t(tile_id) * a.splits + s) * a.tt + c) * size_t(kBM) + row;
#pragma unroll
            for (int j = 0; j < 32; ++j) acc[j] += __ldcg(p + size_t(j) * kBM);
          }
        }
#pragma unroll
        for (int j = 0; j < 32; ++j) v[j] = acc[j];
      }
      epilogue_chunk(a, n, warp, lane, w_tile, tok0 + c, v);
    }
    if (a.splits > 1 && threadIdx.x == 0) a.counters[tile_id] = 0;  // ready for the next launch
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kTmemCols);
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

size_t gemm_scratch_bytes() { return kPartialFloats * sizeof(float) + kCounters * sizeof(int) + 512; }

int make_weight_map(CUtensorMap* map, const void* w, int n_out, int k) {
  return make_map(map, w, k, n_out, kBM);
}

int gemm_run(const GemmProblem& p, const GemmScratch& s, cudaStream_t stream) {
  if (p.n_tok <= 0 || p.n_out <= 0) return SPD_OK;
  if (p.k <= 0) return fail(SPD_EINVAL, "GEMM K must be positive");
  CUtensorMap map_w, map_x;
  const CUtensorMap* mw = p.map_w;
  if (!mw) {
    int rc = make_map(&map_w, p.w, p.k, p.n_out, kBM);
    if (rc) return rc;
    mw = &map_w;
  } else {
    map_w = *mw;
  }
  int rc = make_map(&map_x, p.x, p.k, p.n_tok, kXRows);
  if (rc) return rc;

  KArgs a{};
  a.n_out = p.n_out;
  a.n_tok = p.n_tok;
  a.k = p.k;
  const int n_ttiles = (p.n_tok + 255) / 256;
  a.tt = ((p.n_tok + n_ttiles - 1) / n_ttiles + 31) / 32 * 32;
  a.n_ttiles = n_ttiles;
  a.n_kb = (p.k + kBK - 1) / kBK;
  const int n_wtiles = (p.n_out + kBM - 1) / kBM;
  const int tiles = n_wtiles * n_ttiles;
  const int sms = num_sms();
  // Split K when it fills the SMs noticeably better (at least 4 K blocks per split).
  int best_s = 1;
  double best_eff = 0.0;
  for (int sp = 1; sp <= 16; ++sp) {
    const int kbps = (a.n_kb + sp - 1) / sp;
    const int splits = (a.n_kb + kbps - 1) / kbps;
    if (splits != sp) continue;
    if (sp > 1 && kbps < 4) break;
    if (sp > 1 && size_t(tiles) * sp * a.tt * kBM > s.partial_floats) break;
    if (sp > 1 && tiles > s.n_counters) break;
    const int ctas = tiles * sp;
    const int waves = (ctas + sms - 1) / sms;
    const double eff = double(ctas) / (double(waves) * sms);
    if (eff > best_eff + 0.03) {
      best_eff = eff;
      best_s = sp;
    }
  }
  a.splits = best_s;
  a.kbps = (a.n_kb + best_s - 1) / best_s;
  const int stage_bytes = kWBytes + a.tt * 128;
  a.stages = kSmemPipe / stage_bytes;
  if (a.stages > kMaxStages) a.stages = kMaxStages;
  a.epi = p.epi;
  a.out = p.out;
  a.ldo = p.ldo;
  a.rows = p.rows;
  a.bias = p.bias;
  a.pos = p.pos;
  a.inv_freq = p.inv_freq;
  a.rope_rows = p.rope_rows;
  a.head_dim = p.head_dim;
  a.out_cols = p.out_cols;
  a.partial = s.partial;
  a.counters = s.counters;
  a.status = s.status;
  a.budget = kWaitBudget;

  const size_t smem = size_t(a.stages) * stage_bytes + 1024 + 256;
  static std::once_flag attr_once;
  static cudaError_t attr_err = cudaSuccess;
  std::call_once(attr_once, [] {
    attr_err = cudaFuncSetAttribute(gemm_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                    kSmemPipe + 1024 + 256 + 16384);
  });
  if (attr_err != cudaSuccess)
    return fail(SPD_ECUDA, "cudaFuncSetAttribute: %s", cudaGetErrorString(attr_err));
  dim3 grid(n_ttiles, n_wtiles, a.splits);
  gemm_tc_kernel<<<grid, 128, smem, stream>>>(map_w, map_x, a);
  SPD_CUDA_TRY(cudaGetLastError());
  return SPD_OK;
}

}  // namespace spd
