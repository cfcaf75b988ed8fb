// Variable-length causal attention over packed sequences, queries restricted to the
// attention-active tokens (VSkip-Attn, Sec. 3.2: a skipped token is not a query, but it still
// serves as a key and a value for every other token of its sequence).
//
// One CTA = 64 active queries of one sequence x one head. Four warps own 16 query rows each.
// K/V blocks of 64 keys stream through shared memory (cp.async double buffer). Scores use
// bf16 mma.sync with fp32 accumulation. The softmax is online, in fp32 with exp2, and P is
// rounded to bf16 for the PV product. A query at position p sees keys 0..p of its own sequence.
#include <cuda_bf16.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace spd {
namespace {

constexpr int kQ = 64;   // queries per CTA
constexpr int kKB = 64;  // keys per block

__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(smem))),
               "l"(gmem)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                         uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
      "{%8,%9}, {%0,%1,%2,%3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

template <int HD>
__global__ void __launch_bounds__(128)
    attn_kernel(const __nv_bfloat16* __restrict__ q, int ldq, const __nv_bfloat16* __restrict__ kv,
                int ldkv, int v_off, __nv_bfloat16* __restrict__ o, int ldo,
                const int4* __restrict__ tiles, const int32_t* __restrict__ q_pos, int n_heads,
                int n_kv_heads, float scale_log2) {
  constexpr int LD = HD + 8;  // padded row (elements): conflict-free ldmatrix
  extern __shared__ __align__(16) uint8_t smem_raw[];
  __nv_bfloat16* Qs = reinterpret_cast<__nv_bfloat16*>(smem_raw);
  __nv_bfloat16* Ks = Qs + kQ * LD;
  __nv_bfloat16* Vs = Ks + 2 * kKB * LD;
  int* pos_s = reinterpret_cast<int*>(Vs + 2 * kKB * LD);
  pdl_launch_dependents();
  pdl_wait();

  const int4 tl = tiles[blockIdx.x];
  const int q0 = tl.x, nq = tl.y, kv0 = tl.z;
  const int h = blockIdx.y;
  const int hk = h / (n_heads / n_kv_heads);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = lane >> 2, t4 = lane & 3;

  if (tid < kQ) pos_s[tid] = q_pos[q0 + min(tid, nq - 1)];
  constexpr int CH = HD / 8;  // 16-byte chunks per row
  for (int i = tid; i < kQ * CH; i += 128) {
    const int r = i / CH, c = i % CH;
    const int qr = q0 + min(r, nq - 1);
    cp_async16(Qs + r * LD + c * 8, q + size_t(qr) * ldq + h * HD + c * 8);
  }
  cp_async_commit();
  __syncthreads();
  const int kmax = pos_s[kQ - 1 < nq - 1 ? kQ - 1 : nq - 1] + 1;  // positions ascend in a tile
  const int nkb = (kmax + kKB - 1) / kKB;

  auto load_kv = [&](int kb, int buf) {
    __nv_bfloat16* ks = Ks + buf * kKB * LD;
    __nv_bfloat16* vs = Vs + buf * kKB * LD;
    for (int i = tid; i < kKB * CH; i += 128) {
      const int r = i / CH, c = i % CH;
      const int key = min(kb * kKB + r, kmax - 1);
      const __nv_bfloat16* src = kv + size_t(kv0 + key) * ldkv + hk * HD + c * 8;
      cp_async16(ks + r * LD + c * 8, src);
      cp_async16(vs + r * LD + c * 8, src + v_off);
    }
    cp_async_commit();
  };
  load_kv(0, 0);
  cp_async_wait<1>();
  __syncthreads();

  uint32_t qa[HD / 16][4];
#pragma unroll
  for (int ks = 0; ks < HD / 16; ++ks)
    ldsm_x4(qa[ks], Qs + (warp * 16 + (lane & 15)) * LD + ks * 16 + 8 * (lane >> 4));

  const int p0 = pos_s[warp * 16 + g], p1 = pos_s[warp * 16 + g + 8];
  float oacc[HD / 8][4];
#pragma unroll
  for (int i = 0; i < HD / 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.0f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.0f, l1 = 0.0f;

  for (int kb = 0; kb < nkb; ++kb) {
    const int buf = kb & 1;
    if (kb + 1 < nkb) {
      load_kv(kb + 1, buf ^ 1);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const __nv_bfloat16* ks = Ks + buf * kKB * LD;
    const __nv_bfloat16* vs = Vs + buf * kKB * LD;

    float s[kKB / 8][4];
#pragma unroll
    for (int nt = 0; nt < kKB / 8; ++nt) {
      s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.0f;
#pragma unroll
      for (int ks2 = 0; ks2 < HD / 16; ks2 += 2) {
        uint32_t b[4];
        ldsm_x4(b, ks + (nt * 8 + (lane & 7)) * LD + ks2 * 16 + 8 * (lane >> 3));
        mma16816(s[nt], qa[ks2], b[0], b[1]);
        mma16816(s[nt], qa[ks2 + 1], b[2], b[3]);
      }
    }
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int nt = 0; nt < kKB / 8; ++nt) {
      const int key = kb * kKB + nt * 8 + 2 * t4;
      s[nt][0] = (key <= p0) ? s[nt][0] * scale_log2 : -INFINITY;
      s[nt][1] = (key + 1 <= p0) ? s[nt][1] * scale_log2 : -INFINITY;
      s[nt][2] = (key <= p1) ? s[nt][2] * scale_log2 : -INFINITY;
      s[nt][3] = (key + 1 <= p1) ? s[nt][3] * scale_log2 : -INFINITY;
      mx0 = fmaxf(mx0, fmaxf(s[nt][0], s[nt][1]));
      mx1 = fmaxf(mx1, fmaxf(s[nt][2], s[nt][3]));
    }
#pragma unroll
    for (int off = 1; off <= 2; off <<= 1) {
      mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, off));
      mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, off));
    }
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    const float c0 = exp2f(m0 - mn0), c1 = exp2f(m1 - mn1);  // 0 on the first block (m = -inf)
    m0 = mn0;
    m1 = mn1;
    float rs0 = 0.0f, rs1 = 0.0f;
#pragma unroll
    for (int nt = 0; nt < kKB / 8; ++nt) {
      s[nt][0] = exp2f(s[nt][0] - mn0);
      s[nt][1] = exp2f(s[nt][1] - mn0);
      s[nt][2] = exp2f(s[nt][2] - mn1);
      s[nt][3] = exp2f(s[nt][3] - mn1);
      rs0 += s[nt][0] + s[nt][1];
      rs1 += s[nt][2] + s[nt][3];
    }
    l0 = l0 * c0 + rs0;
    l1 = l1 * c1 + rs1;
#pragma unroll
    for (int i = 0; i < HD / 8; ++i) {
      oacc[i][0] *= c0;
      oacc[i][1] *= c0;
      oacc[i][2] *= c1;
      oacc[i][3] *= c1;
    }
#pragma unroll
    for (int kc = 0; kc < kKB / 16; ++kc) {
      uint32_t pa[4];
      pa[0] = pack_bf16(s[2 * kc][0], s[2 * kc][1]);
      pa[1] = pack_bf16(s[2 * kc][2], s[2 * kc][3]);
      pa[2] = pack_bf16(s[2 * kc + 1][0], s[2 * kc + 1][1]);
      pa[3] = pack_bf16(s[2 * kc + 1][2], s[2 * kc + 1][3]);
#pragma unroll
      for (int nt2 = 0; nt2 < HD / 16; ++nt2) {
        uint32_t b[4];
        ldsm_x4_t(b, vs + (kc * 16 + (lane & 7) + 8 * ((lane >> 3) & 1)) * LD + nt2 * 16 +
                         8 * (lane >> 4));
        mma16816(oacc[2 * nt2], pa, b[0], b[1]);
        mma16816(oacc[2 * nt2 + 1], pa, b[2], b[3]);
      }
    }
    __syncthreads();  // buffer `buf` is refilled by the next iteration's prefetch
  }
#pragma unroll
  for (int off = 1; off <= 2; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  const float i0 = 1.0f / l0, i1 = 1.0f / l1;
  const int r0 = warp * 16 + g, r1 = r0 + 8;
#pragma unroll
  for (int nt = 0; nt < HD / 8; ++nt) {
    const int col = h * HD + nt * 8 + 2 * t4;
    if (r0 < nq)
      *reinterpret_cast<uint32_t*>(o + size_t(q0 + r0) * ldo + col) =
          pack_bf16(oacc[nt][0] * i0, oacc[nt][1] * i0);
    if (r1 < nq)
      *reinterpret_cast<uint32_t*>(o + size_t(q0 + r1) * ldo + col) =
          pack_bf16(oacc[nt][2] * i1, oacc[nt][3] * i1);
  }
}

template <int HD>
int launch(const void* q, int ldq, const void* kv, int ldkv, int v_off, void* o, int ldo,
           const int4* tiles, int n_tiles, const int32_t* q_pos, int n_heads, int n_kv_heads,
           cudaStream_t stream) {
  constexpr int LD = HD + 8;
  const size_t smem = size_t(kQ + 4 * kKB) * LD * 2 + kQ * sizeof(int);
  static bool attr = false;
  if (!attr) {
    SPD_CUDA_TRY(cudaFuncSetAttribute(attn_kernel<HD>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      int(smem)));
    attr = true;
  }
  const float scale_log2 = 1.4426950408889634f / sqrtf(float(HD));
  SPD_CUDA_TRY(launch_pdl(attn_kernel<HD>, dim3(n_tiles, n_heads), dim3(128), smem, stream,
                          static_cast<const __nv_bfloat16*>(q), ldq,
                          static_cast<const __nv_bfloat16*>(kv), ldkv, v_off,
                          static_cast<__nv_bfloat16*>(o), ldo, tiles, q_pos, n_heads, n_kv_heads,
                          scale_log2));
  return SPD_OK;
}

}  // namespace

int attention_run(const void* q, int ldq, const void* kv, int ldkv, int v_off, void* o, int ldo,
                  const int4* tiles, int n_tiles, const int32_t* q_pos, int n_heads, int n_kv_heads,
                  int head_dim, cudaStream_t stream, double ctx_sum, int n_q, int n_kv_rows) {
  if (n_tiles <= 0) return SPD_OK;
  if (head_dim != 128 && head_dim != 64)
    return fail(SPD_EUNSUPPORTED, "attention supports head_dim 64 and 128");
  const int slot = trace_begin(stream);
  const int rc = (head_dim == 128)
                     ? launch<128>(q, ldq, kv, ldkv, v_off, o, ldo, tiles, n_tiles, q_pos, n_heads,
                                   n_kv_heads, stream)
                     : launch<64>(q, ldq, kv, ldkv, v_off, o, ldo, tiles, n_tiles, q_pos, n_heads,
                                  n_kv_heads, stream);
  // QK^T and PV over each active query's causal context; Q, K, V read once and O written once
  trace_end(slot, stream, TR_ATTN, 4.0 * head_dim * n_heads * ctx_sum,
            2.0 * (2.0 * n_q * n_heads * head_dim + 2.0 * n_kv_rows * n_kv_heads * head_dim));
  return rc;
}

}  // namespace spd
