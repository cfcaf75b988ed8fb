// Memory-bound row kernels of the prefill: RMSNorm of the fp32 residual stream into bf16 GEMM
// operands (optionally gathering/scattering rows), bf16 -> fp32 residual initialisation, and bf16
// row scatter for sequence assembly.
#include <cuda_bf16.h>
#include <math.h>
#include <stdint.h>

#include "internal.h"
#include "ptx.cuh"
#include "trace.h"

namespace spd {
namespace {

constexpr int kThreads = 256;

__device__ __forceinline__ float block_sum(float v, float* red) {
#pragma unroll
  for (int off = 16; off; off >>= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = 0.0f;
#pragma unroll
  for (int w = 0; w < kThreads / 32; ++w) t += red[w];
  return t;
}

// out[orow(i)] = bf16(gain * h[irow(i)] / sqrt(mean(h^2) + eps)); out2[map2[irow]] gets the same
// row when map2 is given and map2[irow] >= 0 (compact copy of the attention-active rows). Rows of
// up to kRowVec * 4 * kThreads floats stay in registers between the sum of squares and the scaling
// (one pass over the row); the gains (weights) are loaded before the grid dependency wait.
constexpr int kRowVec = 4;
__device__ __forceinline__ uint2 norm_pack(const float4& v, const ushort4& gg, float inv) {
  const __nv_bfloat162 lo = __floats2bfloat162_rn(
      v.x * inv * __bfloat162float(__ushort_as_bfloat16(gg.x)),
      v.y * inv * __bfloat162float(__ushort_as_bfloat16(gg.y)));
  const __nv_bfloat162 hi = __floats2bfloat162_rn(
      v.z * inv * __bfloat162float(__ushort_as_bfloat16(gg.z)),
      v.w * inv * __bfloat162float(__ushort_as_bfloat16(gg.w)));
  return make_uint2(*reinterpret_cast<const uint32_t*>(&lo), *reinterpret_cast<const uint32_t*>(&hi));
}

__global__ void __launch_bounds__(kThreads)
    rmsnorm_kernel(const float* h, int D, const uint16_t* __restrict__ gain, float eps,
                   const int32_t* in_rows, __nv_bfloat16* __restrict__ out, const int32_t* map2,
                   __nv_bfloat16* __restrict__ out2, unsigned long long* stamp) {
  __shared__ float red[kThreads / 32];
  const int n4 = D / 4;
  const bool in_regs = n4 <= kRowVec * kThreads;
  const ushort4* g4 = reinterpret_cast<const ushort4*>(gain);
  ushort4 gr[kRowVec];
  if (in_regs) {
#pragma unroll
    for (int k = 0; k < kRowVec; ++k) {
      const int c = threadIdx.x + k * kThreads;
      if (c < n4) gr[k] = g4[c];
    }
  }
  pdl_launch_dependents();
  pdl_wait();
  if (threadIdx.x == 0) stamp_start(stamp);
  const int i = blockIdx.x;
  const int r = in_rows ? in_rows[i] : i;
  if (r < 0) return;  // a padding entry of a device-built row list
  const float4* src = reinterpret_cast<const float4*>(h + size_t(r) * D);
  const int r2 = map2 ? map2[r] : -1;
  uint2* o = reinterpret_cast<uint2*>(out + size_t(i) * D);
  uint2* o2 = r2 >= 0 ? reinterpret_cast<uint2*>(out2 + size_t(r2) * D) : nullptr;
  float ss = 0.0f;
  if (in_regs) {
    float4 vr[kRowVec];
#pragma unroll
    for (int k = 0; k < kRowVec; ++k) {
      const int c = threadIdx.x + k * kThreads;
      vr[k] = c < n4 ? src[c] : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < kRowVec; ++k)
      ss += vr[k].x * vr[k].x + vr[k].y * vr[k].y + vr[k].z * vr[k].z + vr[k].w * vr[k].w;
    const float inv = rsqrtf(block_sum(ss, red) / float(D) + eps);
#pragma unroll
    for (int k = 0; k < kRowVec; ++k) {
      const int c = threadIdx.x + k * kThreads;
      if (c < n4) {
        const uint2 pk = norm_pack(vr[k], gr[k], inv);
        o[c] = pk;
        if (o2) o2[c] = pk;
      }
    }
  } else {
    for (int c = threadIdx.x; c < n4; c += kThreads) {
      const float4 v = src[c];
      ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    const float inv = rsqrtf(block_sum(ss, red) / float(D) + eps);
    for (int c = threadIdx.x; c < n4; c += kThreads) {
      const uint2 pk = norm_pack(src[c], g4[c], inv);
      o[c] = pk;
      if (o2) o2[c] = pk;
    }
  }
  if (threadIdx.x == 0) stamp_end(stamp);
}

__global__ void bf16_to_f32_kernel(const uint16_t* x, float* __restrict__ h, size_t n4) {
  pdl_launch_dependents();
  pdl_wait();
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n4;
       i += size_t(gridDim.x) * blockDim.x) {
    const ushort4 v = reinterpret_cast<const ushort4*>(x)[i];
    reinterpret_cast<float4*>(h)[i] =
        make_float4(__uint_as_float(uint32_t(v.x) << 16), __uint_as_float(uint32_t(v.y) << 16),
                    __uint_as_float(uint32_t(v.z) << 16), __uint_as_float(uint32_t(v.w) << 16));
  }
}

__global__ void scatter_rows_kernel(const uint16_t* src, int D, const int32_t* rows,
                                    uint16_t* __restrict__ dst) {
  pdl_launch_dependents();
  pdl_wait();
  const int i = blockIdx.x;
  const uint4* s = reinterpret_cast<const uint4*>(src + size_t(i) * D);
  uint4* d = reinterpret_cast<uint4*>(dst + size_t(rows[i]) * D);
  for (int c = threadIdx.x; c < D / 8; c += blockDim.x) d[c] = s[c];
}

// q_t of sequence b (ASL-Skip's text context, Sec. 4.2.1): the mean of h over the text tokens
// text[ts[b] .. ts[b+1]), one thread per column, tokens in order (zero when there are none).
__global__ void __launch_bounds__(kThreads) text_mean_kernel(const float* h, int D, const int32_t* ts,
                                                             const int32_t* text,
                                                             float* __restrict__ tmean) {
  pdl_launch_dependents();
  pdl_wait();
  const int c = blockIdx.x * kThreads + threadIdx.x, b = blockIdx.y;
  if (c >= D) return;
  const int t0 = ts[b], t1 = ts[b + 1];
  float s = 0.0f;
  for (int e = t0; e < t1; ++e) s += h[size_t(text[e]) * D + c];
  tmean[size_t(b) * D + c] = t1 > t0 ? s / float(t1 - t0) : 0.0f;
}

__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int off = 16; off; off >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, off));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __syncthreads();
  if (lane == 0) red[warp] = v;
  __syncthreads();
  float t = red[0];
#pragma unroll
  for (int w = 1; w < kThreads / 32; ++w) t = fmaxf(t, red[w]);
  return t;
}

// One candidate visual token per CTA (Sec. 4.2.1 and Eq. 6): E_ii = entropy of softmax(logits
// row) / log V, F_itc = (cos(h_i, q_t) + 1) / 2 (0.5 without text), S_sa = ReLU(1 - E - F);
// s_skip[i] += w1 S_sa + w2 SLC^Norm(l), flag[n] = s_skip[i] >= T_skip.
__global__ void __launch_bounds__(kThreads)
    skip_score_kernel(const float* logits, int V, const float* h, int D, const int32_t* cand,
                      const int32_t* ts, const int32_t* seq_of, const float* tmean, float inv_log_v,
                      float w1, float add_slc, float t_skip, int mode, float* s_skip, uint8_t* flag,
                      int32_t* admit, uint8_t* target, int layer, int tgt) {
  __shared__ float red[kThreads / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int n = blockIdx.x, i = cand[n], b = seq_of[i];
  if ((mode & kSkipDevice) && admit[i] >= 0) return;  // already in skip mode (block-uniform)
  float ent = 0.0f;
  if ((mode & kSkipEntropy) && (mode & kSkipLse)) {
    // merge of the per-32-word statistics (m_g, s_g, u_g): with m = max m_g,
    // S = sum_g e^(m_g - m) s_g and U = sum_g e^(m_g - m) (u_g + (m_g - m) s_g), H = log S - U / S
    const int G = lse_groups(V);
    const float4* st = reinterpret_cast<const float4*>(logits) + size_t(n) * G;
    float mx = -INFINITY;
    for (int g = threadIdx.x; g < G; g += kThreads) mx = fmaxf(mx, st[g].x);
    mx = block_max(mx, red);
    float se = 0.0f, te = 0.0f;
    for (int g = threadIdx.x; g < G; g += kThreads) {
      const float4 q = st[g];
      if (q.y > 0.0f) {
        const float dm = q.x - mx, f = expf(dm);
        se += f * q.y;
        te += f * (q.z + dm * q.y);
      }
    }
    __syncthreads();
    se = block_sum(se, red);
    __syncthreads();
    te = block_sum(te, red);
    ent = (logf(se) - te / se) * inv_log_v;
  } else if (mode & kSkipEntropy) {
    const float* z = logits + size_t(n) * V;
    float mx = -INFINITY;
    for (int v = threadIdx.x; v < V; v += kThreads) mx = fmaxf(mx, z[v]);
    mx = block_max(mx, red);
    float se = 0.0f, te = 0.0f;  // sum e^(z - m) and sum e^(z - m) (z - m)
    for (int v = threadIdx.x; v < V; v += kThreads) {
      const float d = z[v] - mx, e = expf(d);
      se += e;
      te += e * d;
    }
    __syncthreads();
    se = block_sum(se, red);
    __syncthreads();
    te = block_sum(te, red);
    ent = (logf(se) - te / se) * inv_log_v;
  }
  const float* hi = h + size_t(i) * D;
  const float* q = tmean + size_t(b) * D;
  float f = 0.0f;
  if (mode & kSkipItc) {
    float dot = 0.0f, hh = 0.0f, qq = 0.0f;
    for (int c = threadIdx.x; c < D; c += kThreads) {
      dot += hi[c] * q[c];
      hh += hi[c] * hi[c];
      qq += q[c] * q[c];
    }
    __syncthreads();
    dot = block_sum(dot, red);
    __syncthreads();
    hh = block_sum(hh, red);
    __syncthreads();
    qq = block_sum(qq, red);
    const bool has_text = ts[b + 1] > ts[b] && hh > 0.0f && qq > 0.0f;
    f = has_text ? 0.5f + 0.5f * dot / (sqrtf(hh) * sqrtf(qq)) : 0.5f;
  }
  if (threadIdx.x == 0) {
    const float s_sa = fmaxf(0.0f, 1.0f - ent - f);
    const float fuse = w1 * s_sa + add_slc;
    const float acc = (mode & kSkipAccumulate) ? s_skip[i] + fuse : fuse;
    s_skip[i] = acc;
    if (mode & kSkipDevice) {
      if (acc >= t_skip) {  // enters skip mode here, its target frozen
        admit[i] = layer;
        target[i] = uint8_t(tgt);
      }
    } else {
      flag[n] = acc >= t_skip ? 1 : 0;
    }
  }
}

// Exclusive prefix sum of one int per thread over the block (blockDim.x a multiple of 32, at most
// 1024); *total receives the block's sum. Every thread must call it.
__device__ int block_scan_excl(int v, int* tmp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
  int x = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, off);
    if (lane >= off) x += y;
  }
  if (lane == 31) tmp[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < nw ? tmp[lane] : 0;
#pragma unroll
    for (int off = 1; off < 32; off <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, off);
      if (lane >= off) w += y;
    }
    tmp[lane] = w;
  }
  __syncthreads();
  const int before = (warp ? tmp[warp - 1] : 0) + x - v;
  *total = tmp[nw - 1];
  __syncthreads();
  return before;
}

// Decoder layer l's row lists from the admission layers, built on the device (the executor's plan
// for a decision made by a kernel): token t bypasses target[t] (1 attention, 2 FFN, 3 both) at
// layer l when 0 <= admit[t] <= l. Outputs in the executor's layout: arows (attention-active
// tokens, ascending; padded to T with -1), amap (token -> its query row or -1), apos (positions of
// the query rows), frows (FFN-active tokens; padded with -1), tiles (up to 128 queries of one
// sequence each; padded to max_tiles with copies of the last tile, whose recomputation writes the
// same values, or a one-query tile when no token is a query). One CTA.
__global__ void __launch_bounds__(1024)
    plan_lists_kernel(int T, int B, const int32_t* cu, const int32_t* pos, const int32_t* admit,
                      const uint8_t* target, int l, const int32_t* kv0, const int32_t* kvlen,
                      int32_t* arows, int32_t* amap, int32_t* apos, int32_t* frows, int4* tiles,
                      int max_tiles) {
  __shared__ int tmp[32];
  __shared__ int seq_cnt[kPlanMaxSeqs];
  pdl_launch_dependents();
  pdl_wait();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  auto bits_of = [&](int t) {
    const int ad = admit[t];
    return (ad >= 0 && ad <= l) ? int(target[t]) : 0;
  };
  int na = 0, nf = 0;
  for (int base = 0; base < T; base += blockDim.x) {
    const int t = base + threadIdx.x;
    const int bits = t < T ? bits_of(t) : 3;
    const int a_act = !(bits & 1), f_act = !(bits & 2);
    int ta, tf;
    const int ea = block_scan_excl(a_act, tmp, &ta);
    const int ef = block_scan_excl(f_act, tmp, &tf);
    if (t < T) {
      if (a_act) {
        arows[na + ea] = t;
        amap[t] = na + ea;
        apos[na + ea] = pos[t];
      } else {
        amap[t] = -1;
      }
      if (f_act) frows[nf + ef] = t;
    }
    na += ta;
    nf += tf;
  }
  for (int r = na + threadIdx.x; r < T; r += blockDim.x) arows[r] = -1;
  for (int r = nf + threadIdx.x; r < T; r += blockDim.x) frows[r] = -1;
  for (int b = warp; b < B; b += blockDim.x >> 5) {  // active queries per sequence
    int cnt = 0;
    for (int t = cu[b] + lane; t < cu[b + 1]; t += 32) cnt += !(bits_of(t) & 1);
#pragma unroll
    for (int off = 16; off; off >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, off);
    if (lane == 0) seq_cnt[b] = cnt;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int a = 0, k = 0;
    for (int b = 0; b < B; ++b) {
      const int n = seq_cnt[b];
      for (int s0 = 0; s0 < n; s0 += 128) tiles[k++] = make_int4(a + s0, min(128, n - s0), kv0[b], kvlen[b]);
      a += n;
    }
    int4 pad;
    if (k > 0) {
      pad = tiles[k - 1];
    } else {
      pad = make_int4(0, 1, kv0[0], kvlen[0]);
      apos[0] = pos[0];
    }
    for (; k < max_tiles; ++k) tiles[k] = pad;
  }
}

}  // namespace

int skip_scores_run(const float* logits, int V, int n_cand, const float* h, int D, const int32_t* cand,
                    const int32_t* ts, const int32_t* text, const int32_t* seq_of, int B, float* tmean,
                    float w1, float add_slc, float t_skip, int mode, float* s_skip, uint8_t* flag,
                    cudaStream_t stream, int32_t* admit, uint8_t* target, int layer, int tgt) {
  if (mode & kSkipItc)
    SPD_CUDA_TRY(launch_pdl(text_mean_kernel, dim3((D + kThreads - 1) / kThreads, B), dim3(kThreads),
                            0, stream, h, D, ts, text, tmean));
  SPD_CUDA_TRY(launch_pdl(skip_score_kernel, dim3(n_cand), dim3(kThreads), 0, stream,
                          logits, V, h, D, cand, ts, seq_of, static_cast<const float*>(tmean),
                          float(1.0 / log(double(V))), w1, add_slc, t_skip, mode, s_skip, flag,
                          admit, target, layer, tgt));
  return SPD_OK;
}

int plan_lists_run(int T, int B, const int32_t* cu, const int32_t* pos, const int32_t* admit,
                   const uint8_t* target, int l, const int32_t* kv0, const int32_t* kvlen,
                   int32_t* arows, int32_t* amap, int32_t* apos, int32_t* frows, int4* tiles,
                   int max_tiles, cudaStream_t stream) {
  if (B > kPlanMaxSeqs) return fail(SPD_EUNSUPPORTED, "device plans support at most %d sequences", kPlanMaxSeqs);
  SPD_CUDA_TRY(launch_pdl(plan_lists_kernel, dim3(1), dim3(1024), 0, stream, T, B, cu, pos, admit,
                          target, l, kv0, kvlen, arows, amap, apos, frows, tiles, max_tiles));
  return SPD_OK;
}

int rmsnorm_run(const float* h, int n_rows, int D, const uint16_t* gain, float eps,
                const int32_t* in_rows, void* out, const int32_t* map2, void* out2,
                cudaStream_t stream) {
  if (n_rows <= 0) return SPD_OK;
  unsigned long long* stamp = stamp_slot(TR_ROWS, 4.0 * n_rows * D, double(n_rows) * D * (4.0 + 2.0));
  const int slot = trace_begin(stream);
  SPD_CUDA_TRY(launch_pdl(rmsnorm_kernel, dim3(n_rows), dim3(kThreads), 0, stream, h, D, gain, eps,
                          in_rows, static_cast<__nv_bfloat16*>(out), map2,
                          static_cast<__nv_bfloat16*>(out2), stamp));
  trace_end(slot, stream, TR_ROWS, 4.0 * n_rows * D, double(n_rows) * D * (4.0 + 2.0));
  return SPD_OK;
}

int bf16_to_f32_run(const uint16_t* x, float* h, size_t n, cudaStream_t stream) {
  if (n == 0) return SPD_OK;
  const size_t n4 = n / 4;
  const int blocks = int((n4 + 255) / 256 < 4096 ? (n4 + 255) / 256 : 4096);
  const int slot = trace_begin(stream);
  SPD_CUDA_TRY(launch_pdl(bf16_to_f32_kernel, dim3(blocks), dim3(256), 0, stream, x, h, n4));
  trace_end(slot, stream, TR_ROWS, 0.0, 6.0 * double(n));
  return SPD_OK;
}

int scatter_rows_run(const uint16_t* src, int n_rows, int D, const int32_t* rows, uint16_t* dst,
                     cudaStream_t stream) {
  if (n_rows <= 0) return SPD_OK;
  const int slot = trace_begin(stream);
  SPD_CUDA_TRY(launch_pdl(scatter_rows_kernel, dim3(n_rows), dim3(128), 0, stream, src, D, rows, dst));
  trace_end(slot, stream, TR_ROWS, 0.0, 4.0 * double(n_rows) * D);
  return SPD_OK;
}

}  // namespace spd
