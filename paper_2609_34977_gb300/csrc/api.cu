// C ABI of libspider.so: errors, model handle (weight re-layout for the GEMM epilogues), skip-plan
// expansion, the projector, and the decoder-prefill executor (Alg. 1 stage 2).
#include <cuda_bf16.h>
#include <math.h>
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <mutex>
#include <memory>
#include <vector>

#include "internal.h"
#include "ptx.cuh"

namespace spd {

int rmsnorm_run(const float* h, int n_rows, int D, const uint16_t* gain, float eps,
                const int32_t* in_rows, void* out, const int32_t* map2, void* out2,
                cudaStream_t stream);
int bf16_to_f32_run(const uint16_t* x, float* h, size_t n, cudaStream_t stream);
int scatter_rows_run(const uint16_t* src, int n_rows, int D, const int32_t* rows, uint16_t* dst,
                     cudaStream_t stream);

static thread_local char g_err[512] = "no error";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int num_sms() {
  int dev = 0, n = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
  return n > 0 ? n : 1;
}

namespace {

// dst[dst_rows[i]][:] = src[src_rows[i]][:] for rows of `cols` bf16.
__global__ void copy_rows_kernel(const uint16_t* __restrict__ src, uint16_t* __restrict__ dst,
                                 int cols, const int32_t* __restrict__ src_rows,
                                 const int32_t* __restrict__ dst_rows, int n) {
  const int i = blockIdx.x;
  if (i >= n) return;
  const uint16_t* s = src + size_t(src_rows[i]) * cols;
  uint16_t* d = dst + size_t(dst_rows[i]) * cols;
  for (int c = threadIdx.x; c < cols; c += blockDim.x) d[c] = s[c];
}

// Bounded wait on a barrier that nothing arrives on: exercises the timeout path.
__global__ void bounded_wait_probe_kernel(int* status, long long budget) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    mbar_init(&bar, 1);
    abort_flag = 0;
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0 && !mbar_wait(&bar, 0, &abort_flag, budget)) set_status(status, SPD_ETIMEOUT);
}

int copy_rows(const void* src, void* dst, int cols, const std::vector<int32_t>& sr,
              const std::vector<int32_t>& dr) {
  if (sr.empty()) return SPD_OK;
  int32_t* d = nullptr;
  SPD_CUDA_TRY(cudaMalloc(&d, sr.size() * 2 * sizeof(int32_t)));
  cudaMemcpy(d, sr.data(), sr.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  cudaMemcpy(d + sr.size(), dr.data(), dr.size() * sizeof(int32_t), cudaMemcpyHostToDevice);
  copy_rows_kernel<<<int(sr.size()), 256>>>(static_cast<const uint16_t*>(src),
                                            static_cast<uint16_t*>(dst), cols, d, d + sr.size(),
                                            int(sr.size()));
  cudaError_t e = cudaDeviceSynchronize();
  cudaFree(d);
  if (e != cudaSuccess) return fail(SPD_ECUDA, "weight packing failed: %s", cudaGetErrorString(e));
  return SPD_OK;
}

// Row order of a Q/K weight inside each head: TMEM lanes l and l + 16 of a warp hold the rotary
// pair (j, j + head_dim/2), so the epilogue rotates with one shuffle.
int rope_source_dim(int r, int hd) {
  const int g = r / 32, l = r % 32;
  return (l < 16) ? 16 * g + l : hd / 2 + 16 * g + (l - 16);
}

}  // namespace
}  // namespace spd

using namespace spd;

struct spd_model {
  spd_model_cfg cfg;
  struct Layer {
    uint16_t *attn_norm, *ffn_norm, *wq, *wkv, *wo, *wgu, *wd;
    CUtensorMap m_qkv, m_kv, m_o, m_gu, m_d;
  };
  std::vector<Layer> layers;
  uint16_t *final_norm = nullptr, *lm_head = nullptr;
  uint16_t *pw1 = nullptr, *pb1 = nullptr, *pw2 = nullptr, *pb2 = nullptr;
  CUtensorMap m_lm, m_p1, m_p2;
  float2* freq = nullptr;  // [head_dim / 2] theta^(-2j / head_dim) in double, split into fp32 (hi, lo)
  int gu_rows = 0;
  void* pool = nullptr;
};

extern "C" const char* spd_last_error(void) { return g_err; }

extern "C" int spd_set_deterministic(int on) {
  set_deterministic(on);
  return SPD_OK;
}

extern "C" int spd_workspace_status(void* ws, void* stream, int* status) {
  if (!ws || !status) return fail(SPD_EINVAL, "null workspace or status");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  int v = 0;
  SPD_CUDA_TRY(cudaMemcpyAsync(&v, ws, sizeof(int), cudaMemcpyDeviceToHost, st));
  SPD_CUDA_TRY(cudaStreamSynchronize(st));
  SPD_CUDA_TRY(cudaMemsetAsync(ws, 0, sizeof(int), st));
  *status = v;
  return SPD_OK;
}

extern "C" int spd_selftest_bounded_wait(void* ws, long long budget_cycles, void* stream) {
  if (!ws) return fail(SPD_EINVAL, "null workspace");
  bounded_wait_probe_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<int*>(ws),
                                                                             budget_cycles);
  SPD_CUDA_TRY(cudaGetLastError());
  return SPD_OK;
}

extern "C" int spd_model_create(const spd_model_cfg* c, const spd_model_weights* w, spd_model** out) {
  if (!c || !w || !out || !w->layers) return fail(SPD_EINVAL, "null model arguments");
  *out = nullptr;
  if (c->n_layers < 1 || c->d_model < 8 || c->n_heads < 1 || c->n_kv_heads < 1 ||
      c->n_heads % c->n_kv_heads || c->d_ffn < 8 || c->vocab < 1)
    return fail(SPD_EINVAL, "invalid model shape");
  if (c->head_dim != 64 && c->head_dim != 128)
    return fail(SPD_EUNSUPPORTED, "head_dim must be 64 or 128");
  if (c->d_model % 8 || c->d_ffn % 8 || (c->d_vis && (c->d_vis % 8 || c->d_proj % 8 || c->d_proj < 8)))
    return fail(SPD_EINVAL, "d_model, d_ffn, d_vis, d_proj must be multiples of 8");
  if ((c->n_heads * c->head_dim) % 128 || (c->n_kv_heads * c->head_dim) % 128)
    return fail(SPD_EUNSUPPORTED, "heads * head_dim must be a multiple of 128");
  const size_t D = c->d_model, F = c->d_ffn, hd = c->head_dim;
  const size_t q_rows = c->n_heads * hd, kv_rows = c->n_kv_heads * hd;
  const int gu_rows = int((F + 63) / 64 * 128);
  auto al = [](size_t b) { return (b + 255) & ~size_t(255); };
  const size_t per_layer = al(D * 2) * 2 + al(q_rows * D * 2) + al(2 * kv_rows * D * 2) +
                           al(D * q_rows * 2) + al(size_t(gu_rows) * D * 2) + al(D * F * 2);
  size_t total = per_layer * c->n_layers + al(D * 2) + al(size_t(c->vocab) * D * 2) + al(hd * 8);
  if (c->d_vis)
    total += al(size_t(c->d_proj) * c->d_vis * 2) + al(size_t(c->d_proj) * 2) +
             al(D * c->d_proj * 2) + al(D * 2);
  spd_model* m = new spd_model();
  m->cfg = *c;
  m->gu_rows = gu_rows;
  if (cudaMalloc(&m->pool, total) != cudaSuccess) {
    delete m;
    return fail(SPD_ECUDA, "cudaMalloc of %zu bytes for the model failed", total);
  }
  cudaMemset(m->pool, 0, total);
  uint8_t* cur = static_cast<uint8_t*>(m->pool);
  auto take = [&](size_t b) {
    uint8_t* p = cur;
    cur += al(b);
    return reinterpret_cast<uint16_t*>(p);
  };
  int rc = SPD_OK;
  auto fin = [&](int code) {
    if (code) {
      cudaFree(m->pool);
      delete m;
    }
    return code;
  };
  std::vector<int32_t> sr, dr;
  m->layers.resize(c->n_layers);
  for (int l = 0; l < c->n_layers && !rc; ++l) {
    const spd_layer_weights& s = w->layers[l];
    spd_model::Layer& L = m->layers[l];
    if (!s.attn_norm || !s.wq || !s.wk || !s.wv || !s.wo || !s.ffn_norm || !s.w_gate || !s.w_up ||
        !s.w_down)
      return fin(fail(SPD_EINVAL, "null weight in layer %d", l));
    L.attn_norm = take(D * 2);
    L.ffn_norm = take(D * 2);
    L.wq = take(q_rows * D * 2);
    L.wkv = take(2 * kv_rows * D * 2);
    L.wo = take(D * q_rows * 2);
    L.wgu = take(size_t(gu_rows) * D * 2);
    L.wd = take(D * F * 2);
    cudaMemcpy(L.attn_norm, s.attn_norm, D * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(L.ffn_norm, s.ffn_norm, D * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(L.wo, s.wo, D * q_rows * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(L.wd, s.w_down, D * F * 2, cudaMemcpyDeviceToDevice);
    // Q rows in rotary-pair order
    sr.clear();
    dr.clear();
    for (size_t r = 0; r < q_rows; ++r) {
      dr.push_back(int32_t(r));
      sr.push_back(int32_t((r / hd) * hd + rope_source_dim(int(r % hd), int(hd))));
    }
    if ((rc = copy_rows(s.wq, L.wq, int(D), sr, dr))) break;
    // K rows in rotary-pair order, then V rows as they are
    sr.clear();
    dr.clear();
    for (size_t r = 0; r < kv_rows; ++r) {
      dr.push_back(int32_t(r));
      sr.push_back(int32_t((r / hd) * hd + rope_source_dim(int(r % hd), int(hd))));
    }
    if ((rc = copy_rows(s.wk, L.wkv, int(D), sr, dr))) break;
    cudaMemcpy(L.wkv + kv_rows * D, s.wv, kv_rows * D * 2, cudaMemcpyDeviceToDevice);
    // gate/up interleaved in half-warps: 128-row tile i, row 32 w + l holds gate (l < 16) or up
    // (l >= 16) of FFN channel 64 i + 16 w + (l mod 16)
    std::vector<int32_t> gs, gd, us, ud;
    for (int r = 0; r < gu_rows; ++r) {
      const int tile = r / 128, w32 = (r % 128) / 32, l32 = r % 32;
      const int f = tile * 64 + w32 * 16 + (l32 & 15);
      if (f >= int(F)) continue;
      if (l32 < 16) { gs.push_back(f); gd.push_back(r); }
      else { us.push_back(f); ud.push_back(r); }
    }
    if ((rc = copy_rows(s.w_gate, L.wgu, int(D), gs, gd))) break;
    if ((rc = copy_rows(s.w_up, L.wgu, int(D), us, ud))) break;
    if (L.wkv != L.wq + q_rows * D) {  // the pool keeps them adjacent (sizes multiples of 256 B)
      rc = fail(SPD_EUNSUPPORTED, "Wq and Wk|Wv are not adjacent");
      break;
    }
    if ((rc = make_weight_map(&L.m_qkv, L.wq, int(q_rows + 2 * kv_rows), int(D)))) break;
    if ((rc = make_weight_map(&L.m_kv, L.wkv, int(2 * kv_rows), int(D)))) break;
    if ((rc = make_weight_map(&L.m_o, L.wo, int(D), int(q_rows)))) break;
    if ((rc = make_weight_map(&L.m_gu, L.wgu, gu_rows, int(D)))) break;
    if ((rc = make_weight_map(&L.m_d, L.wd, int(D), int(F)))) break;
  }
  if (rc) return fin(rc);
  if (!w->final_norm || !w->lm_head) return fin(fail(SPD_EINVAL, "null final_norm or lm_head"));
  m->final_norm = take(D * 2);
  m->lm_head = take(size_t(c->vocab) * D * 2);
  cudaMemcpy(m->final_norm, w->final_norm, D * 2, cudaMemcpyDeviceToDevice);
  cudaMemcpy(m->lm_head, w->lm_head, size_t(c->vocab) * D * 2, cudaMemcpyDeviceToDevice);
  if ((rc = make_weight_map(&m->m_lm, m->lm_head, c->vocab, int(D)))) return fin(rc);
  m->freq = reinterpret_cast<float2*>(take(hd / 2 * sizeof(float2)));
  std::vector<float2> fr(hd / 2);
  for (size_t j = 0; j < hd / 2; ++j) {
    const double f = pow(double(c->rope_theta), -2.0 * double(j) / double(hd));
    const float hi = float(f);
    fr[j] = make_float2(hi, float(f - double(hi)));
  }
  cudaMemcpy(m->freq, fr.data(), fr.size() * sizeof(float2), cudaMemcpyHostToDevice);
  if (c->d_vis) {
    if (!w->proj_w1 || !w->proj_b1 || !w->proj_w2 || !w->proj_b2)
      return fin(fail(SPD_EINVAL, "null projector weight"));
    m->pw1 = take(size_t(c->d_proj) * c->d_vis * 2);
    m->pb1 = take(size_t(c->d_proj) * 2);
    m->pw2 = take(D * c->d_proj * 2);
    m->pb2 = take(D * 2);
    cudaMemcpy(m->pw1, w->proj_w1, size_t(c->d_proj) * c->d_vis * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(m->pb1, w->proj_b1, size_t(c->d_proj) * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(m->pw2, w->proj_w2, D * c->d_proj * 2, cudaMemcpyDeviceToDevice);
    cudaMemcpy(m->pb2, w->proj_b2, D * 2, cudaMemcpyDeviceToDevice);
    if ((rc = make_weight_map(&m->m_p1, m->pw1, c->d_proj, c->d_vis))) return fin(rc);
    if ((rc = make_weight_map(&m->m_p2, m->pw2, int(D), c->d_proj))) return fin(rc);
  }
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return fin(fail(SPD_ECUDA, "model upload: %s", cudaGetErrorString(e)));
  *out = m;
  return SPD_OK;
}

extern "C" void spd_model_destroy(spd_model* m) {
  if (!m) return;
  cudaFree(m->pool);
  delete m;
}

extern "C" int spd_plan_adaptive(int n_layers, int n_tokens, const int16_t* admit,
                                 const uint8_t* target, uint8_t* mask) {
  if (n_layers < 1 || n_tokens < 0 || (n_tokens && (!admit || !target)) || !mask)
    return fail(SPD_EINVAL, "bad plan arguments");
  memset(mask, 0, size_t(n_layers) * n_tokens);
  for (int i = 0; i < n_tokens; ++i) {
    if (admit[i] < 0) continue;
    if (target[i] < 1 || target[i] > 3) return fail(SPD_EINVAL, "token %d: target must be 1, 2 or 3", i);
    for (int l = admit[i]; l < n_layers; ++l) mask[size_t(l) * n_tokens + i] = target[i];
  }
  return SPD_OK;
}

extern "C" int spd_plan_static(int n_layers, int n_tokens, const uint8_t* layer_mask,
                               const uint8_t* token_sel, uint8_t* mask) {
  if (n_layers < 1 || n_tokens < 0 || !layer_mask || (n_tokens && !token_sel) || !mask)
    return fail(SPD_EINVAL, "bad plan arguments");
  for (int l = 0; l < n_layers; ++l) {
    if (layer_mask[l] > 3) return fail(SPD_EINVAL, "layer %d: mask bits must be in 0..3", l);
    for (int i = 0; i < n_tokens; ++i)
      mask[size_t(l) * n_tokens + i] = token_sel[i] ? layer_mask[l] : 0;
  }
  return SPD_OK;
}

// ---- linear (single GEMM) --------------------------------------------------------------------
extern "C" size_t spd_linear_workspace_size(int, int) { return 256 + gemm_scratch_bytes(); }

static GemmScratch scratch_from(Carve& cv) {
  GemmScratch s;
  s.partial_floats = kGemmSlotFloats;
  s.partial = cv.take<float>(s.partial_floats);
  s.n_counters = 1 << 16;
  s.counters = cv.take<int>(s.n_counters);
  s.acc = nullptr;
  s.acc_floats = 0;
  s.status = cv.status();
  return s;
}
// The accumulation buffers, carved last in a workspace (after the activation buffers).
static void take_acc(Carve& cv, GemmScratch& s) {
  s.acc_floats = kGemmAccFloats;
  s.acc = cv.take<float>(s.acc_floats);
}

extern "C" int spd_linear(const uint16_t* X, int M, int K, const uint16_t* W, int N, int epilogue,
                          const uint16_t* bias, const int32_t* rows, void* out, int ldo, void* ws,
                          size_t ws_bytes, void* stream) {
  if (!X || !W || !out || !ws || M < 0 || K < 8 || N < 1 || ldo < N)
    return fail(SPD_EINVAL, "bad linear arguments");
  if (epilogue < SPD_EPI_F32 || epilogue > SPD_EPI_ADD_F32) return fail(SPD_EINVAL, "bad epilogue");
  if ((epilogue == SPD_EPI_BIAS_BF16 || epilogue == SPD_EPI_BIAS_GELU_BF16) && !bias)
    return fail(SPD_EINVAL, "epilogue needs a bias");
  Carve cv(ws, ws_bytes);
  GemmScratch s = scratch_from(cv);
  take_acc(cv, s);
  if (!cv.fits()) return fail(SPD_ENOSPC, "linear workspace too small");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (int rc = gemm_scratch_clear(s, st)) return rc;
  GemmProblem p{};
  p.w = W;
  p.x = X;
  p.n_out = N;
  p.n_tok = M;
  p.k = K;
  p.epi = epilogue;
  p.out = out;
  p.ldo = ldo;
  p.rows = rows;
  p.bias = bias;
  p.out_cols = N;
  return gemm_run(p, s, st);
}

// ---- allocation-free variant of spd_linear ---------------------------------------------------
// Scratch of spd_linear_noalloc: status word, per-tile counters, then partial-sum slots.
static __device__ __align__(256) uint8_t g_linear_scratch[SPD_LINEAR_NOALLOC_SCRATCH_BYTES];

namespace {
constexpr int kMaxDevices = 64;
std::mutex g_linear_scratch_mu;
void* g_linear_scratch_ptr[kMaxDevices] = {};  // per device, set by the first call on it

// Address of g_linear_scratch on the current device, looked up once per device.
int linear_scratch(void** out) {
  int dev = 0;
  SPD_CUDA_TRY(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kMaxDevices) return fail(SPD_EUNSUPPORTED, "device ordinal %d", dev);
  std::lock_guard<std::mutex> lock(g_linear_scratch_mu);
  if (!g_linear_scratch_ptr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_linear_scratch);
    if (e != cudaSuccess) return fail(SPD_ECUDA, "cudaGetSymbolAddress: %s", cudaGetErrorString(e));
    g_linear_scratch_ptr[dev] = p;
  }
  *out = g_linear_scratch_ptr[dev];
  return SPD_OK;
}
}  // namespace

extern "C" int spd_linear_noalloc(const uint16_t* X, int M, int K, const uint16_t* W, int N,
                                  int epilogue, const uint16_t* bias, const int32_t* rows, void* out,
                                  int ldo, int* status, void* stream) {
  if (!X || !W || !out || M < 0 || K < 8 || N < 1 || ldo < N)
    return fail(SPD_EINVAL, "bad linear arguments");
  if (epilogue < SPD_EPI_F32 || epilogue > SPD_EPI_ADD_F32) return fail(SPD_EINVAL, "bad epilogue");
  if ((epilogue == SPD_EPI_BIAS_BF16 || epilogue == SPD_EPI_BIAS_GELU_BF16) && !bias)
    return fail(SPD_EINVAL, "epilogue needs a bias");
  // tile counters of the worst tiling gemm_run may choose: CTA pairs count each 128-row half of a
  // 256-row tile (2 ceil(N / 256) >= ceil(N / 128) per token tile of 256)
  const long long tiles = 2LL * ((N + 255) / 256) * ((M + 255) / 256);
  if (tiles > SPD_LINEAR_NOALLOC_MAX_TILES)
    return fail(SPD_ENOSPC, "spd_linear_noalloc: %lld tile counters exceed the static scratch (%d)",
                tiles, SPD_LINEAR_NOALLOC_MAX_TILES);
  void* base = nullptr;
  if (int rc = linear_scratch(&base)) return rc;
  Carve cv(base, SPD_LINEAR_NOALLOC_SCRATCH_BYTES);
  GemmScratch s;
  s.status = cv.status();
  s.n_counters = SPD_LINEAR_NOALLOC_MAX_TILES;
  s.counters = cv.take<int>(s.n_counters);
  s.partial = cv.take<float>(0);
  s.partial_floats = (SPD_LINEAR_NOALLOC_SCRATCH_BYTES - cv.used) / sizeof(float);
  s.acc = nullptr;  // no accumulation buffers: stream-K partial slots only
  s.acc_floats = 0;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // the status word and the counters start at zero (a failed earlier call may have left them set)
  SPD_CUDA_TRY(cudaMemsetAsync(base, 0, 256, st));
  if (int rc = gemm_scratch_clear(s, st)) return rc;
  GemmProblem p{};
  p.w = W;
  p.x = X;
  p.n_out = N;
  p.n_tok = M;
  p.k = K;
  p.epi = epilogue;
  p.out = out;
  p.ldo = ldo;
  p.rows = rows;
  p.bias = bias;
  p.out_cols = N;
  if (int rc = gemm_run(p, s, st)) return rc;
  if (status) SPD_CUDA_TRY(cudaMemcpyAsync(status, s.status, sizeof(int), cudaMemcpyDeviceToDevice, st));
  return SPD_OK;
}

// ---- projector and sequence assembly --------------------------------------------------------
extern "C" size_t spd_project_workspace_size(const spd_model* m, int rows) {
  if (!m || rows < 0) return 0;
  Carve cv(nullptr, ~size_t(0));
  GemmScratch s = scratch_from(cv);
  cv.take<uint16_t>(size_t(rows) * (m->cfg.d_proj > 0 ? m->cfg.d_proj : 1));
  take_acc(cv, s);
  return cv.used;
}

extern "C" int spd_project(const spd_model* m, const uint16_t* vis, int rows, const int32_t* out_rows,
                           uint16_t* x, void* ws, size_t ws_bytes, void* stream) {
  if (!m || !vis || !out_rows || !x || !ws || rows < 0) return fail(SPD_EINVAL, "bad project arguments");
  if (!m->cfg.d_vis) return fail(SPD_EINVAL, "model has no projector");
  Carve cv(ws, ws_bytes);
  GemmScratch s = scratch_from(cv);
  uint16_t* hid = cv.take<uint16_t>(size_t(rows) * m->cfg.d_proj);
  take_acc(cv, s);
  if (!cv.fits()) return fail(SPD_ENOSPC, "project workspace too small");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (int rc = gemm_scratch_clear(s, st)) return rc;
  GemmProblem p{};
  p.map_w = &m->m_p1;
  p.w = m->pw1;
  p.x = vis;
  p.n_out = m->cfg.d_proj;
  p.n_tok = rows;
  p.k = m->cfg.d_vis;
  p.epi = EPI_BIAS_GELU_BF16;
  p.out = hid;
  p.ldo = m->cfg.d_proj;
  p.bias = m->pb1;
  if (int rc = gemm_run(p, s, st)) return rc;
  p.map_w = &m->m_p2;
  p.w = m->pw2;
  p.x = hid;
  p.n_out = m->cfg.d_model;
  p.k = m->cfg.d_proj;
  p.epi = EPI_BIAS_BF16;
  p.out = x;
  p.ldo = m->cfg.d_model;
  p.bias = m->pb2;
  p.rows = out_rows;
  return gemm_run(p, s, st);
}

extern "C" int spd_scatter_rows(const spd_model* m, const uint16_t* src, int rows,
                                const int32_t* rows_map, uint16_t* dst, void* stream) {
  if (!m || !src || !rows_map || !dst || rows < 0) return fail(SPD_EINVAL, "bad scatter arguments");
  return scatter_rows_run(src, rows, m->cfg.d_model, rows_map, dst, static_cast<cudaStream_t>(stream));
}

// ---- attention on its own ---------------------------------------------------------------------
namespace {
size_t attention_tiles(int n_q, int n_seqs) { return size_t(n_q) / kAttnTileQ + n_seqs + 1; }
}  // namespace

extern "C" size_t spd_attention_workspace_size(int n_q, int n_seqs) {
  if (n_q < 1 || n_seqs < 1) return 0;
  Carve cv(nullptr, ~size_t(0));
  cv.take<int4>(attention_tiles(n_q, n_seqs));
  return cv.used;
}

extern "C" int spd_attention(const uint16_t* q, int n_q, const int32_t* q_pos, const int32_t* q_cu,
                             const uint16_t* kv, int n_kv, const int32_t* cu, int B, int n_heads,
                             int n_kv_heads, int head_dim, uint16_t* o, void* ws, size_t ws_bytes,
                             void* stream) {
  if (!q || !q_pos || !q_cu || !kv || !cu || !o || !ws || n_q < 1 || n_kv < 1 || B < 1 ||
      n_heads < 1 || n_kv_heads < 1 || n_heads % n_kv_heads)
    return fail(SPD_EINVAL, "bad attention arguments");
  if (q_cu[0] != 0 || q_cu[B] != n_q || cu[0] != 0 || cu[B] != n_kv)
    return fail(SPD_EINVAL, "q_cu and cu_seqlens must run from 0 to n_q and n_kv");
  for (int b = 0; b < B; ++b)
    if (q_cu[b + 1] < q_cu[b] || cu[b + 1] <= cu[b] || q_cu[b + 1] - q_cu[b] > cu[b + 1] - cu[b])
      return fail(SPD_EINVAL, "sequence %d: empty, decreasing, or more queries than tokens", b);
  Carve cv(ws, ws_bytes);
  int4* tiles = cv.take<int4>(attention_tiles(n_q, B));
  if (!cv.fits()) return fail(SPD_ENOSPC, "attention workspace too small");
  std::vector<int4> ht;
  for (int b = 0; b < B; ++b)
    for (int s0 = q_cu[b]; s0 < q_cu[b + 1]; s0 += kAttnTileQ)
      ht.push_back(make_int4(s0, std::min(kAttnTileQ, q_cu[b + 1] - s0), cu[b], cu[b + 1] - cu[b]));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  SPD_CUDA_TRY(cudaMemcpyAsync(tiles, ht.data(), ht.size() * sizeof(int4), cudaMemcpyHostToDevice, st));
  const int kvd = n_kv_heads * head_dim;
  double ctx = 0.0;  // for the trace only: an upper bound (every key of the sequence)
  for (int b = 0; b < B; ++b) ctx += double(q_cu[b + 1] - q_cu[b]) * (cu[b + 1] - cu[b]);
  return attention_run(q, n_q, kv, n_kv, 2 * kvd, kvd, o, n_heads * head_dim, tiles, int(ht.size()),
                       q_pos, n_heads, n_kv_heads, head_dim, cv.status(), st, ctx);
}

// ---- prefill executor ------------------------------------------------------------------------
namespace {

struct PrefillBufs {
  uint16_t *xa, *q, *kv, *o, *y, *act, *z;
  int32_t* lists;
  size_t list_ints;
  GemmScratch gs;
};

// Every list starts on a multiple of 4 ints (16 bytes): the attention tiles are read as int4.
size_t pad4(size_t n) { return (n + 3) & ~size_t(3); }
size_t list_ints_for(int L, int T, int B) {
  // per layer: arows[T], amap[T], apos[T], frows[T], tiles[(T / 64 + B + 1) * 4]
  // plus pos_all[T], kvrow[T], last[B]
  return size_t(L) * (4 * pad4(T) + 4 * (size_t(T) / 64 + B + 1)) + 2 * pad4(T) + pad4(B) + 16;
}

PrefillBufs carve_prefill(const spd_model_cfg& c, int T, int B, Carve& cv) {
  PrefillBufs b;
  const size_t D = c.d_model, qd = size_t(c.n_heads) * c.head_dim, kvd = size_t(c.n_kv_heads) * c.head_dim;
  b.gs = scratch_from(cv);
  b.xa = cv.take<uint16_t>(size_t(T) * D);
  b.q = cv.take<uint16_t>(size_t(T) * qd);
  b.kv = cv.take<uint16_t>(size_t(T) * 2 * kvd);
  b.o = cv.take<uint16_t>(size_t(T) * qd);
  b.y = cv.take<uint16_t>(size_t(T) * D);
  b.act = cv.take<uint16_t>(size_t(T) * c.d_ffn);
  b.z = cv.take<uint16_t>(size_t(B) * D);
  b.list_ints = list_ints_for(c.n_layers, T, B);
  b.lists = cv.take<int32_t>(b.list_ints);
  take_acc(cv, b.gs);
  return b;
}

}  // namespace

extern "C" size_t spd_prefill_workspace_size(const spd_model* m, int max_tokens, int max_seqs) {
  if (!m || max_tokens < 1 || max_seqs < 1) return 0;
  Carve cv(nullptr, ~size_t(0));
  carve_prefill(m->cfg, max_tokens, max_seqs, cv);
  return cv.used;
}

namespace {

// Host side of one prefill call: the per-layer row lists (the plan is control data: it decides
// which launches happen), in one int32 buffer whose layout the device copy shares.
struct LayerLists {
  size_t arows, amap, apos, frows, tiles;  // offsets into the buffer
  int na, nf, ntiles;
  double ctx;
};
struct HostPlan {
  std::vector<int32_t> hl;
  std::vector<int> pos_all, seq_of;
  std::vector<int> kv0, kvlen;  // per sequence: first key row and key count of its attention
  std::vector<LayerLists> ll;
  size_t pos_off = 0, kvrow_off = 0, last_off = 0, end = 0;
  bool decode = false;  // one query per sequence at its last position (attention_decode_run)
};

// Token t of sequence b = seq_of at position pos_all; its K/V row is kvrow (cache modes) or t.
// Sequence b attends over key rows [kv0[b], kv0[b] + kvlen[b]).
void plan_init(HostPlan& P, const spd_model_cfg& c, const int32_t* cu, int B, int T, size_t list_ints,
               const int* pos = nullptr, int max_len = 0) {
  P.hl.assign(list_ints, 0);
  P.pos_all.assign(T, 0);
  P.seq_of.assign(T, 0);
  P.kv0.assign(B, 0);
  P.kvlen.assign(B, 0);
  for (int b = 0; b < B; ++b) {
    for (int t = cu[b]; t < cu[b + 1]; ++t) {
      P.pos_all[t] = (pos ? pos[b] : 0) + t - cu[b];
      P.seq_of[t] = b;
    }
    P.kv0[b] = max_len ? b * max_len : cu[b];
    P.kvlen[b] = (pos ? pos[b] : 0) + cu[b + 1] - cu[b];
  }
  P.ll.assign(c.n_layers, LayerLists{});
  P.decode = false;
  size_t off = 0;
  P.pos_off = off;
  for (int t = 0; t < T; ++t) P.hl[off + t] = P.pos_all[t];
  off += pad4(T);
  P.kvrow_off = off;
  for (int t = 0; t < T; ++t) P.hl[off + t] = max_len ? P.seq_of[t] * max_len + P.pos_all[t] : t;
  off += pad4(T);
  P.last_off = off;
  for (int b = 0; b < B; ++b) P.hl[off + b] = cu[b + 1] - 1;
  off += pad4(B);
  for (int l = 0; l < c.n_layers; ++l) {
    LayerLists& q = P.ll[l];
    q.arows = off; off += pad4(T);
    q.amap = off; off += pad4(T);
    q.apos = off; off += pad4(T);
    q.frows = off; off += pad4(T);
    q.tiles = off;
    off += 4 * (size_t(T) / 64 + B + 1);
  }
  P.end = off;
}

// Layer l's lists from its skip bits (bit 0 skip attention, bit 1 skip FFN; null = none).
void plan_layer(HostPlan& P, int l, const uint8_t* mk, const int32_t* cu, int B, int T) {
  LayerLists& q = P.ll[l];
  std::vector<int32_t>& hl = P.hl;
  q.na = q.nf = q.ntiles = 0;
  q.ctx = 0.0;
  for (int t = 0; t < T; ++t) {
    const int bits = mk ? mk[t] : 0;
    if (!(bits & 1)) {
      hl[q.amap + t] = q.na;
      hl[q.apos + q.na] = P.pos_all[t];
      q.ctx += P.pos_all[t] + 1;
      hl[q.arows + q.na++] = t;
    } else {
      hl[q.amap + t] = -1;
    }
    if (!(bits & 2)) hl[q.frows + q.nf++] = t;
  }
  // attention tiles: up to kAttnTileQ active queries of one sequence each
  int a = 0;
  for (int b = 0; b < B; ++b) {
    int a_end = a;
    while (a_end < q.na && P.seq_of[hl[q.arows + a_end]] == b) ++a_end;
    for (int s0 = a; s0 < a_end; s0 += kAttnTileQ) {
      int32_t* tl = &hl[q.tiles + 4 * size_t(q.ntiles++)];
      tl[0] = s0;
      tl[1] = (a_end - s0 < kAttnTileQ) ? a_end - s0 : kAttnTileQ;
      tl[2] = P.kv0[b];
      tl[3] = P.kvlen[b];
    }
    a = a_end;
  }
}

int validate_prefill(const spd_model* m, const uint16_t* x, int T, const int32_t* cu, int B,
                     const float* h, const void* ws) {
  if (!m || !x || !cu || !h || !ws || T < 1 || B < 1) return fail(SPD_EINVAL, "bad prefill arguments");
  if (cu[0] != 0 || cu[B] != T) return fail(SPD_EINVAL, "cu_seqlens must run from 0 to n_tokens");
  for (int b = 0; b < B; ++b)
    if (cu[b + 1] <= cu[b]) return fail(SPD_EINVAL, "sequence %d is empty or cu_seqlens decreases", b);
  return SPD_OK;
}

// Where layer l's K and V go: the prefill's scratch (rows = tokens) or a cache block.
struct KVDest {
  uint16_t* kv;  // [n_rows][2 kvd]
  int n_rows;
  bool cache;    // rows from the plan's kvrow list
};

// Decoder layer l on the residual stream h with its lists at dl (device copy of the plan).
int run_layer(const spd_model* m, int l, const LayerLists& q, const HostPlan& P, const PrefillBufs& bf,
              const int32_t* dl, float* h, int T, cudaStream_t st, const KVDest* kvd_dest = nullptr) {
  const spd_model_cfg& c = m->cfg;
  const int D = c.d_model, hd = c.head_dim;
  const int qd = c.n_heads * hd, kvd = c.n_kv_heads * hd;
  const spd_model::Layer& W = m->layers[l];
  int rc;
  // attention sub-layer: norm of every row (K/V need all tokens); one GEMM gives K, V of every
  // token and Q of the query tokens (rows of skipped tokens computed but not stored: the
  // contraction is weight-bound, one pass over Wq|Wk|Wv beats two launches). On the
  // matrix-vector path (a few tokens) the GEMM applies the norm itself.
  const KVDest dest = kvd_dest ? *kvd_dest : KVDest{bf.kv, T, false};
  const int32_t* kvrow = dest.cache ? dl + P.kvrow_off : nullptr;
  GemmProblem kvp{};
  kvp.map_w = &W.m_kv;
  kvp.w = W.wkv;
  kvp.x = bf.xa;
  kvp.n_out = 2 * kvd;
  kvp.n_tok = T;
  kvp.k = D;
  kvp.epi = EPI_ROPE_BF16;
  kvp.out = dest.kv;
  kvp.ldo = 2 * kvd;
  kvp.rows = kvrow;
  kvp.pos = dl + P.pos_off;
  kvp.rope = m->freq;
  kvp.rope_rows = kvd;
  kvp.head_dim = hd;
  auto with_norm = [&](GemmProblem& p, const uint16_t* gain, const int32_t* rows, int n,
                       void* xbuf) -> int {
    if (gemm_fuses_norm(p)) {
      p.norm_h = h;
      p.norm_gain = gain;
      p.norm_rows = rows;
      p.norm_eps = c.rms_eps;
      return SPD_OK;
    }
    return rmsnorm_run(h, n, D, gain, c.rms_eps, rows, xbuf, nullptr, nullptr, st);
  };
  if (q.na > 0) {
    GemmProblem qp = kvp;
    qp.map_w = &W.m_qkv;
    qp.w = W.wq;  // Wq rows, then Wk and Wv rows, contiguous
    qp.n_out = qd + 2 * kvd;
    qp.epi = EPI_QKV_BF16;
    qp.out = bf.q;
    qp.ldo = qd;
    qp.rows = dl + q.amap;
    qp.out2 = dest.kv;
    qp.rows2 = kvrow;
    qp.ldo2 = 2 * kvd;
    qp.split = qd;
    qp.n_tok_out = q.na;
    if ((rc = with_norm(qp, W.attn_norm, nullptr, T, bf.xa))) return rc;
    if ((rc = gemm_run(qp, bf.gs, st))) return rc;
  } else {
    if ((rc = with_norm(kvp, W.attn_norm, nullptr, T, bf.xa))) return rc;
    if ((rc = gemm_run(kvp, bf.gs, st))) return rc;
  }
  if (q.na > 0) {
    if (P.decode)
      rc = attention_decode_run(bf.q, dest.kv, 2 * kvd, kvd, bf.o, qd,
                                reinterpret_cast<const int4*>(dl + q.tiles), q.ntiles, c.n_heads,
                                c.n_kv_heads, hd, st, q.ctx);
    else
      rc = attention_run(bf.q, q.na, dest.kv, dest.n_rows, 2 * kvd, kvd, bf.o, qd,
                         reinterpret_cast<const int4*>(dl + q.tiles), q.ntiles, dl + q.apos,
                         c.n_heads, c.n_kv_heads, hd, bf.gs.status, st, q.ctx);
    if (rc) return rc;
    GemmProblem op{};
    op.map_w = &W.m_o;
    op.w = W.wo;
    op.x = bf.o;
    op.n_out = D;
    op.n_tok = q.na;
    op.k = qd;
    op.epi = EPI_ADD_F32;
    op.out = h;
    op.ldo = D;
    op.rows = dl + q.arows;
    if ((rc = gemm_run(op, bf.gs, st))) return rc;
  }
  if (q.nf > 0) {
    GemmProblem gp{};
    gp.map_w = &W.m_gu;
    gp.w = W.wgu;
    gp.x = bf.y;
    gp.n_out = m->gu_rows;
    gp.n_tok = q.nf;
    gp.k = D;
    gp.epi = EPI_SWIGLU_BF16;
    gp.out = bf.act;
    gp.ldo = c.d_ffn;
    gp.out_cols = c.d_ffn;
    if ((rc = with_norm(gp, W.ffn_norm, dl + q.frows, q.nf, bf.y))) return rc;
    if ((rc = gemm_run(gp, bf.gs, st))) return rc;
    GemmProblem dp{};
    dp.map_w = &W.m_d;
    dp.w = W.wd;
    dp.x = bf.act;
    dp.n_out = D;
    dp.n_tok = q.nf;
    dp.k = c.d_ffn;
    dp.epi = EPI_ADD_F32;
    dp.out = h;
    dp.ldo = D;
    dp.rows = dl + q.frows;
    if ((rc = gemm_run(dp, bf.gs, st))) return rc;
  }
  return SPD_OK;
}

// Final norm and LM head of each sequence's last token.
int run_head(const spd_model* m, const HostPlan& P, const PrefillBufs& bf, const int32_t* dl,
             float* h, int B, float* logits, cudaStream_t st) {
  if (!logits) return SPD_OK;
  const spd_model_cfg& c = m->cfg;
  GemmProblem lp{};
  lp.map_w = &m->m_lm;
  lp.w = m->lm_head;
  lp.x = bf.z;
  lp.n_out = c.vocab;
  lp.n_tok = B;
  lp.k = c.d_model;
  lp.epi = EPI_F32;
  lp.out = logits;
  lp.ldo = c.vocab;
  if (gemm_fuses_norm(lp)) {  // the final norm of the last tokens, inside the matrix-vector kernel
    lp.norm_h = h;
    lp.norm_gain = m->final_norm;
    lp.norm_rows = dl + P.last_off;
    lp.norm_eps = c.rms_eps;
  } else if (int rc = rmsnorm_run(h, B, c.d_model, m->final_norm, c.rms_eps, dl + P.last_off, bf.z,
                                  nullptr, nullptr, st)) {
    return rc;
  }
  return gemm_run(lp, bf.gs, st);
}

}  // namespace

extern "C" int spd_prefill(const spd_model* m, const uint16_t* x, int T, const int32_t* cu, int B,
                           const uint8_t* mask, float* h, float* logits, void* ws, size_t ws_bytes,
                           void* stream) {
  if (int rc = validate_prefill(m, x, T, cu, B, h, ws)) return rc;
  if (mask)
    for (size_t i = 0; i < size_t(m->cfg.n_layers) * T; ++i)
      if (mask[i] > 3) return fail(SPD_EINVAL, "skip mask entries must be in 0..3");
  const spd_model_cfg& c = m->cfg;
  Carve cv(ws, ws_bytes);
  PrefillBufs bf = carve_prefill(c, T, B, cv);
  if (!cv.fits()) return fail(SPD_ENOSPC, "prefill workspace too small (%zu < %zu)", ws_bytes, cv.used);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  static thread_local HostPlan P;
  plan_init(P, c, cu, B, T, bf.list_ints);
  for (int l = 0; l < c.n_layers; ++l) plan_layer(P, l, mask ? mask + size_t(l) * T : nullptr, cu, B, T);
  int32_t* dl = bf.lists;
  SPD_CUDA_TRY(cudaMemcpyAsync(dl, P.hl.data(), P.end * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  if (int rc = gemm_scratch_clear(bf.gs, st)) return rc;
  if (int rc = bf16_to_f32_run(x, h, size_t(T) * c.d_model, st)) return rc;
  for (int l = 0; l < c.n_layers; ++l)
    if (int rc = run_layer(m, l, P.ll[l], P, bf, dl, h, T, st)) return rc;
  return run_head(m, P, bf, dl, h, B, logits, st);
}

// ---- prefill with the online ASL-Skip plan (Alg. 1 stage 2) -----------------------------------
namespace {
struct AdaptiveBufs {
  float* logits;  // [T][lse_groups(V)] float4 logit-lens statistics of the candidates
  float* tmean;   // [B][D] mean text hidden state per sequence
  float* s_skip;  // [T] accumulated skippability
  uint8_t* flag;  // [T] admitted at this layer (per candidate)
  int32_t* cand;  // [T] candidate token indices
  int32_t* seq;   // [T] sequence of every token
  int32_t* ts;    // [B + 1] text-token ranges
  int32_t* text;  // [T] text-token indices
  // device plan
  int32_t* admit;   // [T] admission layer (-1 = never)
  uint8_t* target;  // [T] frozen target
  int32_t* cu;      // [B + 1]
  int32_t* kv0;     // [B] first key row of each sequence
  int32_t* kvlen;   // [B] key count of each sequence
};
AdaptiveBufs carve_adaptive(const spd_model_cfg& c, int T, int B, Carve& cv) {
  AdaptiveBufs a;
  a.logits = cv.take<float>(size_t(T) * lse_groups(c.vocab) * 4);
  a.tmean = cv.take<float>(size_t(B) * c.d_model);
  a.s_skip = cv.take<float>(T);
  a.flag = cv.take<uint8_t>(T);
  a.cand = cv.take<int32_t>(T);
  a.seq = cv.take<int32_t>(T);
  a.ts = cv.take<int32_t>(B + 1);
  a.text = cv.take<int32_t>(T);
  a.admit = cv.take<int32_t>(T);
  a.target = cv.take<uint8_t>(T);
  a.cu = cv.take<int32_t>(B + 1);
  a.kv0 = cv.take<int32_t>(B);
  a.kvlen = cv.take<int32_t>(B);
  return a;
}
}  // namespace

extern "C" size_t spd_prefill_adaptive_workspace_size(const spd_model* m, int max_tokens, int max_seqs) {
  if (!m || max_tokens < 1 || max_seqs < 1) return 0;
  Carve cv(nullptr, ~size_t(0));
  carve_prefill(m->cfg, max_tokens, max_seqs, cv);
  carve_adaptive(m->cfg, max_tokens, max_seqs, cv);
  return cv.used;
}

extern "C" int spd_prefill_adaptive(const spd_model* m, const uint16_t* x, int T, const int32_t* cu,
                                    int B, const spd_skip_policy* pol, int16_t* admit_layer,
                                    float* h, float* logits, void* ws, size_t ws_bytes,
                                    void* stream) {
  if (int rc = validate_prefill(m, x, T, cu, B, h, ws)) return rc;
  if (!pol || !pol->slc_norm || !pol->layer_target || !pol->is_visual || !admit_layer)
    return fail(SPD_EINVAL, "adaptive prefill needs a policy (SLC^Norm, targets, visual tokens)");
  const spd_model_cfg& c = m->cfg;
  const int L = c.n_layers, D = c.d_model;
  if (pol->window < 0 || pol->window > L) return fail(SPD_EINVAL, "window must lie in [0, n_layers]");
  for (int l = 0; l < L; ++l)
    if (pol->layer_target[l] != 1 && pol->layer_target[l] != 2)
      return fail(SPD_EINVAL, "layer targets must be 1 (attention) or 2 (FFN)");
  const int ab_bits = SPD_SKIP_NO_ENTROPY | SPD_SKIP_NO_ITC | SPD_SKIP_NO_ACCUM | SPD_SKIP_NO_SLC;
  if (pol->ablate & ~ab_bits) return fail(SPD_EINVAL, "unknown ablate bits");
  // which parts of Eq. 4-6 run (S_sa's terms are not computed where w1 = 0 makes them irrelevant)
  const bool no_slc = pol->ablate & SPD_SKIP_NO_SLC;
  const int mode = ((pol->w1 != 0.0f && !(pol->ablate & SPD_SKIP_NO_ENTROPY)) ? kSkipEntropy : 0) |
                   ((pol->w1 != 0.0f && !(pol->ablate & SPD_SKIP_NO_ITC)) ? kSkipItc : 0) |
                   ((pol->ablate & SPD_SKIP_NO_ACCUM) ? 0 : kSkipAccumulate) | kSkipLse;
  Carve cv(ws, ws_bytes);
  PrefillBufs bf = carve_prefill(c, T, B, cv);
  AdaptiveBufs ab = carve_adaptive(c, T, B, cv);
  if (!cv.fits()) return fail(SPD_ENOSPC, "adaptive prefill workspace too small (%zu < %zu)", ws_bytes, cv.used);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  static thread_local HostPlan P;
  plan_init(P, c, cu, B, T, bf.list_ints);
  int32_t* dl = bf.lists;
  // positions and last tokens; sequences and text tokens of the scores
  SPD_CUDA_TRY(cudaMemcpyAsync(dl, P.hl.data(), (P.ll.empty() ? P.end : P.ll[0].arows) * sizeof(int32_t),
                               cudaMemcpyHostToDevice, st));
  std::vector<int32_t> seq(P.seq_of.begin(), P.seq_of.end()), ts(B + 1, 0), text;
  for (int b = 0; b < B; ++b) {
    for (int t = cu[b]; t < cu[b + 1]; ++t)
      if (!pol->is_visual[t]) text.push_back(t);
    ts[b + 1] = int32_t(text.size());
  }
  SPD_CUDA_TRY(cudaMemcpyAsync(ab.seq, seq.data(), T * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  SPD_CUDA_TRY(cudaMemcpyAsync(ab.ts, ts.data(), (B + 1) * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  if (!text.empty())
    SPD_CUDA_TRY(cudaMemcpyAsync(ab.text, text.data(), text.size() * sizeof(int32_t),
                                 cudaMemcpyHostToDevice, st));
  SPD_CUDA_TRY(cudaMemsetAsync(ab.s_skip, 0, T * sizeof(float), st));
  if (int rc = gemm_scratch_clear(bf.gs, st)) return rc;
  if (int rc = bf16_to_f32_run(x, h, size_t(T) * D, st)) return rc;

  // logit lens of nc candidate tokens (device list): final RMSNorm, then the unembedding with the
  // entropy's statistics taken in the GEMM's epilogue (per 32 vocabulary words: max, sum of
  // exponentials and their weighted sum; the fp32 logits never reach memory)
  auto lens = [&](const int32_t* cand_dev, int nc) -> int {
    if (int rc = rmsnorm_run(h, nc, D, m->final_norm, c.rms_eps, cand_dev, bf.xa, nullptr, nullptr, st))
      return rc;
    GemmProblem up{};
    up.map_w = &m->m_lm;
    up.w = m->lm_head;
    up.x = bf.xa;
    up.n_out = c.vocab;
    up.n_tok = nc;
    up.k = D;
    up.epi = EPI_LSE_F32;
    up.out = ab.logits;
    up.ldo = lse_groups(c.vocab);
    return gemm_run(up, bf.gs, st);
  };

  if (pol->device_plan) {
    // Decisions and row lists on the device: every window layer scores every visual token (those
    // already in skip mode are passed over), admits on the device, and a kernel rebuilds the row
    // lists; the sub-layers then run over all T rows with the lists' padding rows skipped. No
    // host round trip until the admission layers are read back at the end.
    std::vector<int32_t> vis;
    for (int t = 0; t < T; ++t)
      if (pol->is_visual[t]) vis.push_back(t);
    const int nv = int(vis.size());
    if (nv > 0)
      SPD_CUDA_TRY(cudaMemcpyAsync(ab.cand, vis.data(), nv * sizeof(int32_t), cudaMemcpyHostToDevice, st));
    std::vector<int32_t> kv0(P.kv0.begin(), P.kv0.end()), kvl(P.kvlen.begin(), P.kvlen.end());
    SPD_CUDA_TRY(cudaMemcpyAsync(ab.cu, cu, (B + 1) * sizeof(int32_t), cudaMemcpyHostToDevice, st));
    SPD_CUDA_TRY(cudaMemcpyAsync(ab.kv0, kv0.data(), B * sizeof(int32_t), cudaMemcpyHostToDevice, st));
    SPD_CUDA_TRY(cudaMemcpyAsync(ab.kvlen, kvl.data(), B * sizeof(int32_t), cudaMemcpyHostToDevice, st));
    SPD_CUDA_TRY(cudaMemsetAsync(ab.admit, 0xff, T * sizeof(int32_t), st));  // -1: never
    SPD_CUDA_TRY(cudaMemsetAsync(ab.target, 0, T, st));
    // Each decision layer writes its own list block; the layers past the window reuse the last
    // decision layer's block.
    int max_tiles = 0;
    for (int b = 0; b < B; ++b) max_tiles += (cu[b + 1] - cu[b] + kAttnTileQ - 1) / kAttnTileQ;
    double ctx_all = 0.0;
    for (int t = 0; t < T; ++t) ctx_all += P.pos_all[t] + 1;
    const int last_block = pol->window > 0 ? pol->window - 1 : 0;
    for (int l = 0; l < L; ++l) {
      LayerLists LD = P.ll[l < last_block ? l : last_block];
      LD.na = T;
      LD.nf = T;
      LD.ntiles = max_tiles;
      LD.ctx = ctx_all;
      if (l < pol->window && nv > 0) {
        if (mode & kSkipEntropy)
          if (int rc = lens(ab.cand, nv)) return rc;
        const float add_slc = no_slc ? 0.0f : pol->w2 * pol->slc_norm[l];
        if (int rc = skip_scores_run(ab.logits, c.vocab, nv, h, D, ab.cand, ab.ts, ab.text, ab.seq, B,
                                     ab.tmean, pol->w1, add_slc, pol->t_skip, mode | kSkipDevice,
                                     ab.s_skip, ab.flag, st, ab.admit, ab.target, l,
                                     no_slc ? 3 : pol->layer_target[l]))
          return rc;
      }
      if (l <= last_block)  // past the window the plan no longer changes
        if (int rc = plan_lists_run(T, B, ab.cu, dl + P.pos_off, ab.admit, ab.target, l, ab.kv0,
                                    ab.kvlen, dl + LD.arows, dl + LD.amap, dl + LD.apos, dl + LD.frows,
                                    reinterpret_cast<int4*>(dl + LD.tiles), max_tiles, st))
          return rc;
      if (int rc = run_layer(m, l, LD, P, bf, dl, h, T, st)) return rc;
    }
    std::vector<int32_t> ad(T);
    SPD_CUDA_TRY(cudaMemcpyAsync(ad.data(), ab.admit, T * sizeof(int32_t), cudaMemcpyDeviceToHost, st));
    const int rc = run_head(m, P, bf, dl, h, B, logits, st);
    SPD_CUDA_TRY(cudaStreamSynchronize(st));
    for (int t = 0; t < T; ++t) admit_layer[t] = int16_t(ad[t]);
    return rc;
  }

  std::vector<int> admit(T, -1);
  std::vector<uint8_t> target(T, 0), row(T, 0), flags(T);
  std::vector<int32_t> cand;
  for (int l = 0; l < L; ++l) {
    if (l < pol->window) {
      // the decision before layer l's forward, on its input hidden states (Alg. 1)
      cand.clear();
      for (int t = 0; t < T; ++t)
        if (pol->is_visual[t] && admit[t] < 0) cand.push_back(t);
      const int nc = int(cand.size());
      if (nc > 0) {
        SPD_CUDA_TRY(cudaMemcpyAsync(ab.cand, cand.data(), nc * sizeof(int32_t),
                                     cudaMemcpyHostToDevice, st));
        if (mode & kSkipEntropy)
          if (int rc = lens(ab.cand, nc)) return rc;
        const float add_slc = no_slc ? 0.0f : pol->w2 * pol->slc_norm[l];
        if (int rc = skip_scores_run(ab.logits, c.vocab, nc, h, D, ab.cand, ab.ts, ab.text, ab.seq, B,
                                     ab.tmean, pol->w1, add_slc, pol->t_skip, mode, ab.s_skip, ab.flag,
                                     st))
          return rc;
        SPD_CUDA_TRY(cudaMemcpyAsync(flags.data(), ab.flag, nc, cudaMemcpyDeviceToHost, st));
        SPD_CUDA_TRY(cudaStreamSynchronize(st));
        for (int n = 0; n < nc; ++n)
          if (flags[n]) {
            admit[cand[n]] = l;
            target[cand[n]] = no_slc ? 3 : pol->layer_target[l];  // frozen at admission
          }
      }
    }
    for (int t = 0; t < T; ++t) row[t] = (admit[t] >= 0 && admit[t] <= l) ? target[t] : 0;
    plan_layer(P, l, row.data(), cu, B, T);
    const LayerLists& q = P.ll[l];
    const size_t blk_end = q.tiles + 4 * (size_t(T) / 64 + B + 1);
    SPD_CUDA_TRY(cudaMemcpyAsync(dl + q.arows, P.hl.data() + q.arows, (blk_end - q.arows) * sizeof(int32_t),
                                 cudaMemcpyHostToDevice, st));
    if (int rc = run_layer(m, l, q, P, bf, dl, h, T, st)) return rc;
  }
  for (int t = 0; t < T; ++t) admit_layer[t] = int16_t(admit[t]);
  return run_head(m, P, bf, dl, h, B, logits, st);
}

// ---- KV cache and decode (the cache a prefill leaves for generation) --------------------------
extern "C" size_t spd_kv_cache_bytes(const spd_model* m, int n_seqs, int max_len) {
  if (!m || n_seqs < 1 || max_len < 1) return 0;
  return size_t(m->cfg.n_layers) * n_seqs * max_len * 2 * m->cfg.n_kv_heads * m->cfg.head_dim *
         sizeof(uint16_t);
}

extern "C" int spd_prefill_kv(const spd_model* m, const uint16_t* x, int T, const int32_t* cu, int B,
                              const uint8_t* mask, float* h, float* logits, uint16_t* kv_cache,
                              int max_len, void* ws, size_t ws_bytes, void* stream) {
  if (int rc = validate_prefill(m, x, T, cu, B, h, ws)) return rc;
  if (!kv_cache || max_len < 1) return fail(SPD_EINVAL, "null KV cache or max_len < 1");
  for (int b = 0; b < B; ++b)
    if (cu[b + 1] - cu[b] > max_len) return fail(SPD_EINVAL, "sequence %d is longer than max_len", b);
  if (mask)
    for (size_t i = 0; i < size_t(m->cfg.n_layers) * T; ++i)
      if (mask[i] > 3) return fail(SPD_EINVAL, "skip mask entries must be in 0..3");
  const spd_model_cfg& c = m->cfg;
  Carve cv(ws, ws_bytes);
  PrefillBufs bf = carve_prefill(c, T, B, cv);
  if (!cv.fits()) return fail(SPD_ENOSPC, "prefill workspace too small (%zu < %zu)", ws_bytes, cv.used);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  static thread_local HostPlan P;
  plan_init(P, c, cu, B, T, bf.list_ints, nullptr, max_len);
  for (int l = 0; l < c.n_layers; ++l) plan_layer(P, l, mask ? mask + size_t(l) * T : nullptr, cu, B, T);
  int32_t* dl = bf.lists;
  SPD_CUDA_TRY(cudaMemcpyAsync(dl, P.hl.data(), P.end * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  if (int rc = gemm_scratch_clear(bf.gs, st)) return rc;
  if (int rc = bf16_to_f32_run(x, h, size_t(T) * c.d_model, st)) return rc;
  const size_t layer_rows = size_t(B) * max_len, row = 2 * size_t(c.n_kv_heads) * c.head_dim;
  for (int l = 0; l < c.n_layers; ++l) {
    const KVDest dest{kv_cache + l * layer_rows * row, int(layer_rows), true};
    if (int rc = run_layer(m, l, P.ll[l], P, bf, dl, h, T, st, &dest)) return rc;
  }
  return run_head(m, P, bf, dl, h, B, logits, st);
}

namespace {
size_t carve_decode(const spd_model_cfg& c, int B, Carve& cv, PrefillBufs* bf, float** h) {
  *bf = carve_prefill(c, B, B, cv);
  *h = cv.take<float>(size_t(B) * c.d_model);
  return cv.used;
}
}  // namespace

extern "C" size_t spd_decode_workspace_size(const spd_model* m, int n_seqs) {
  if (!m || n_seqs < 1) return 0;
  Carve cv(nullptr, ~size_t(0));
  PrefillBufs bf;
  float* h;
  return carve_decode(m->cfg, n_seqs, cv, &bf, &h);
}

extern "C" int spd_decode(const spd_model* m, const uint16_t* x, int B, const int32_t* pos,
                          uint16_t* kv_cache, int max_len, float* logits, void* ws, size_t ws_bytes,
                          void* stream) {
  if (!m || !x || !pos || !kv_cache || !logits || !ws || B < 1 || max_len < 1)
    return fail(SPD_EINVAL, "bad decode arguments");
  for (int b = 0; b < B; ++b)
    if (pos[b] < 0 || pos[b] >= max_len) return fail(SPD_EINVAL, "position of sequence %d outside [0, max_len)", b);
  const spd_model_cfg& c = m->cfg;
  Carve cv(ws, ws_bytes);
  PrefillBufs bf;
  float* h;
  carve_decode(c, B, cv, &bf, &h);
  if (!cv.fits()) return fail(SPD_ENOSPC, "decode workspace too small (%zu < %zu)", ws_bytes, cv.used);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  std::vector<int32_t> cu(B + 1);
  for (int b = 0; b <= B; ++b) cu[b] = b;
  static thread_local HostPlan P;
  plan_init(P, c, cu.data(), B, B, bf.list_ints, pos, max_len);
  P.decode = true;
  for (int l = 0; l < c.n_layers; ++l) plan_layer(P, l, nullptr, cu.data(), B, B);
  int32_t* dl = bf.lists;
  SPD_CUDA_TRY(cudaMemcpyAsync(dl, P.hl.data(), P.end * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  if (int rc = gemm_scratch_clear(bf.gs, st)) return rc;
  if (int rc = bf16_to_f32_run(x, h, size_t(B) * c.d_model, st)) return rc;
  const size_t layer_rows = size_t(B) * max_len, row = 2 * size_t(c.n_kv_heads) * c.head_dim;
  for (int l = 0; l < c.n_layers; ++l) {
    const KVDest dest{kv_cache + l * layer_rows * row, int(layer_rows), true};
    if (int rc = run_layer(m, l, P.ll[l], P, bf, dl, h, B, st, &dest)) return rc;
  }
  return run_head(m, P, bf, dl, h, B, logits, st);
}


// ---- the hot path's contract names (thin forms of the calls above) --------------------------------
extern "C" size_t spd_prune_workspace(const spd_prune_cfg* cfg) { return spd_prune_workspace_size(cfg); }

extern "C" size_t spd_prefill_workspace(const spd_model* m, int total_tokens, int n_seqs) {
  return spd_prefill_workspace_size(m, total_tokens, n_seqs);
}

extern "C" int spd_gather_bf16(const float* payload, int n_tok, const int32_t* keep_idx, int n_tiles,
                               int keep, int has_cls, int d, uint16_t* out, void* stream) {
  return spd_gather_rows_bf16(payload, n_tiles, n_tok, d, has_cls ? 1 : 0, keep_idx, keep, out, nullptr,
                              stream);
}

extern "C" int spd_last_error_detail(char* buf, size_t n) {
  const char* msg = spd_last_error();
  const size_t len = strlen(msg);
  if (buf && n > 0) {
    const size_t c = len < n - 1 ? len : n - 1;
    memcpy(buf, msg, c);
    buf[c] = '\0';
  }
  return int(len);
}

extern "C" int spd_check(void* ws, void* stream) {
  int status = SPD_OK;
  if (int rc = spd_workspace_status(ws, stream, &status)) return rc;
  return status;
}

extern "C" int spd_plan_from_layer_mask(int n_layers, int n_tokens, const uint8_t* layer_mask,
                                        const uint8_t* token_is_visual, uint8_t* mask) {
  return spd_plan_static(n_layers, n_tokens, layer_mask, token_is_visual, mask);
}

extern "C" int spd_prefill_admit(const spd_model* m, const uint16_t* x, int T, const int32_t* cu, int B,
                                 const int16_t* admit_layer, const uint8_t* target, float* h,
                                 float* logits, void* ws, size_t ws_bytes, void* stream) {
  if (!admit_layer && !target) return spd_prefill(m, x, T, cu, B, nullptr, h, logits, ws, ws_bytes, stream);
  if (!m || !admit_layer || !target || T < 1) return fail(SPD_EINVAL, "admit_layer and target go together");
  std::vector<uint8_t> mask(size_t(m->cfg.n_layers) * T);
  if (int rc = spd_plan_adaptive(m->cfg.n_layers, T, admit_layer, target, mask.data())) return rc;
  return spd_prefill(m, x, T, cu, B, mask.data(), h, logits, ws, ws_bytes, stream);
}

// ---- one whole SPIDER step through the C ABI (host or device buffers) ------------------------------
namespace {
bool on_host(const void* p) {
  cudaPointerAttributes at{};
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    cudaGetLastError();
    return true;  // unknown to CUDA: pageable host memory
  }
  return at.type == cudaMemoryTypeHost || at.type == cudaMemoryTypeUnregistered;
}

struct StepLayout {
  int B = 0, T = 0, n_tiles = 0, n_vis = 0, n_text = 0, n_patch = 0;
  std::vector<int32_t> cu, vis_rows, text_rows;
};

int step_layout(const spd_model* m, const spd_prune_cfg* pc, int B, const int32_t* tiles_per_seq,
                const int32_t* text_len, StepLayout* L) {
  if (!m || !pc || B < 1 || !tiles_per_seq || !text_len) return fail(SPD_EINVAL, "bad step arguments");
  L->B = B;
  L->n_patch = pc->n_tok - (pc->has_cls ? 1 : 0);
  L->cu.assign(1, 0);
  L->vis_rows.clear();
  L->text_rows.clear();
  int row = 0, tiles = 0;
  for (int b = 0; b < B; ++b) {
    if (tiles_per_seq[b] < 0 || text_len[b] < 0 || tiles_per_seq[b] + text_len[b] == 0)
      return fail(SPD_EINVAL, "sequence %d: negative or empty", b);
    const int nv = tiles_per_seq[b] * pc->keep;
    for (int i = 0; i < nv; ++i) L->vis_rows.push_back(row++);
    for (int i = 0; i < text_len[b]; ++i) L->text_rows.push_back(row++);
    L->cu.push_back(row);
    tiles += tiles_per_seq[b];
  }
  if (tiles != pc->n_tiles) return fail(SPD_EINVAL, "tiles_per_seq sums to %d, cfg.n_tiles is %d", tiles, pc->n_tiles);
  L->T = row;
  L->n_tiles = tiles;
  L->n_vis = int(L->vis_rows.size());
  L->n_text = int(L->text_rows.size());
  if (!m->cfg.d_vis && pc->d_feat != m->cfg.d_model)
    return fail(SPD_EINVAL, "without a projector the feature width must equal d_model");
  if (m->cfg.d_vis && pc->d_feat != m->cfg.d_vis) return fail(SPD_EINVAL, "feature width != projector input");
  return SPD_OK;
}

// Carves the step's buffers; sizes only when base is null.
struct StepBufs {
  const float* feats[SPD_MAX_FEAT_LAYERS];
  float *feat_copy[SPD_MAX_FEAT_LAYERS], *attn_copy, *logits_dev;
  uint16_t *text_copy, *vis, *x;
  float* h;
  int32_t *keep_idx, *rows;  // rows: vis_rows then text_rows
  uint8_t *prune_ws, *proj_ws, *pre_ws;
  size_t prune_bytes, proj_bytes, pre_bytes;
};
size_t step_carve(const spd_model* m, const spd_prune_cfg* pc, const StepLayout& L, void* base,
                  StepBufs* s) {
  Carve cv(base, ~size_t(0));
  const size_t tile = size_t(pc->n_tok) * pc->d_feat;
  for (int l = 0; l < pc->n_layers; ++l) s->feat_copy[l] = cv.take<float>(size_t(pc->n_tiles) * tile);
  const int n_att = pc->attn_form == 0 ? pc->n_tok : L.n_patch;
  s->attn_copy = cv.take<float>(size_t(pc->n_tiles) * pc->n_heads * n_att);
  s->text_copy = cv.take<uint16_t>(size_t(L.n_text) * m->cfg.d_model);
  s->logits_dev = cv.take<float>(size_t(L.B) * m->cfg.vocab);
  s->keep_idx = cv.take<int32_t>(size_t(pc->n_tiles) * pc->keep);
  s->rows = cv.take<int32_t>(size_t(L.n_vis + L.n_text));
  s->vis = cv.take<uint16_t>(size_t(L.n_vis) * pc->d_feat);
  s->x = cv.take<uint16_t>(size_t(L.T) * m->cfg.d_model);
  s->h = cv.take<float>(size_t(L.T) * m->cfg.d_model);
  s->prune_bytes = spd_prune_workspace_size(pc);
  s->prune_ws = cv.take<uint8_t>(s->prune_bytes);
  s->proj_bytes = m->cfg.d_vis ? spd_project_workspace_size(m, L.n_vis) : 0;
  s->proj_ws = cv.take<uint8_t>(s->proj_bytes);
  s->pre_bytes = spd_prefill_workspace_size(m, L.T, L.B);
  s->pre_ws = cv.take<uint8_t>(s->pre_bytes);
  return cv.used;
}
}  // namespace

extern "C" size_t spd_step_workspace_size(const spd_model* m, const spd_prune_cfg* cfg, int n_seqs,
                                          const int32_t* tiles_per_seq, const int32_t* text_len) {
  StepLayout L;
  if (step_layout(m, cfg, n_seqs, tiles_per_seq, text_len, &L)) return 0;
  if (!spd_prune_workspace_size(cfg)) return 0;
  StepBufs s;
  return step_carve(m, cfg, L, nullptr, &s);
}

extern "C" int spd_step(const spd_model* m, const spd_prune_cfg* cfg, int n_seqs,
                        const int32_t* tiles_per_seq, const int32_t* text_len,
                        const float* const* feats, const float* attn, const uint16_t* text,
                        const uint8_t* skip_mask, float* logits, void* ws, size_t ws_bytes, void* stream) {
  StepLayout L;
  if (int rc = step_layout(m, cfg, n_seqs, tiles_per_seq, text_len, &L)) return rc;
  if (!feats || !attn || (L.n_text && !text) || !logits || !ws) return fail(SPD_EINVAL, "null step buffer");
  if (cfg->n_layers < 1 || cfg->n_layers > SPD_MAX_FEAT_LAYERS) return fail(SPD_EINVAL, "bad feature layer count");
  StepBufs s;
  const size_t need = step_carve(m, cfg, L, ws, &s);
  if (need > ws_bytes) return fail(SPD_ENOSPC, "step workspace too small (%zu < %zu)", ws_bytes, need);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const size_t tile = size_t(cfg->n_tok) * cfg->d_feat;
  // inputs in host memory are copied into the workspace first
  for (int l = 0; l < cfg->n_layers; ++l) {
    if (!feats[l]) return fail(SPD_EINVAL, "null feature layer %d", l);
    s.feats[l] = feats[l];
    if (on_host(feats[l])) {
      SPD_CUDA_TRY(cudaMemcpyAsync(s.feat_copy[l], feats[l], cfg->n_tiles * tile * sizeof(float),
                                   cudaMemcpyHostToDevice, st));
      s.feats[l] = s.feat_copy[l];
    }
  }
  const int n_att = cfg->attn_form == 0 ? cfg->n_tok : L.n_patch;
  const float* attn_d = attn;
  if (on_host(attn)) {
    SPD_CUDA_TRY(cudaMemcpyAsync(s.attn_copy, attn, size_t(cfg->n_tiles) * cfg->n_heads * n_att * sizeof(float),
                                 cudaMemcpyHostToDevice, st));
    attn_d = s.attn_copy;
  }
  const uint16_t* text_d = text;
  const size_t D = m->cfg.d_model;
  if (L.n_text && on_host(text)) {
    SPD_CUDA_TRY(cudaMemcpyAsync(s.text_copy, text, L.n_text * D * sizeof(uint16_t), cudaMemcpyHostToDevice, st));
    text_d = s.text_copy;
  }
  std::vector<int32_t> rows(L.vis_rows);
  rows.insert(rows.end(), L.text_rows.begin(), L.text_rows.end());
  if (!rows.empty())
    SPD_CUDA_TRY(cudaMemcpyAsync(s.rows, rows.data(), rows.size() * sizeof(int32_t), cudaMemcpyHostToDevice, st));
  // MSV-Prune, gather, projector (or row copy), text rows, prefill
  if (int rc = spd_prune(cfg, s.feats, attn_d, s.keep_idx, nullptr, nullptr, nullptr, s.prune_ws, s.prune_bytes,
                         stream))
    return rc;
  if (int rc = spd_gather_rows_bf16(s.feats[cfg->final_layer], cfg->n_tiles, cfg->n_tok, cfg->d_feat,
                                    cfg->has_cls ? 1 : 0, s.keep_idx, cfg->keep, s.vis, s.prune_ws, stream))
    return rc;
  if (L.n_vis) {
    const int rc = m->cfg.d_vis ? spd_project(m, s.vis, L.n_vis, s.rows, s.x, s.proj_ws, s.proj_bytes, stream)
                                : spd_scatter_rows(m, s.vis, L.n_vis, s.rows, s.x, stream);
    if (rc) return rc;
  }
  if (L.n_text)
    if (int rc = spd_scatter_rows(m, text_d, L.n_text, s.rows + L.n_vis, s.x, stream)) return rc;
  const bool host_logits = on_host(logits);
  float* lg = host_logits ? s.logits_dev : logits;
  if (int rc = spd_prefill(m, s.x, L.T, L.cu.data(), L.B, skip_mask, s.h, lg, s.pre_ws, s.pre_bytes, stream))
    return rc;
  if (host_logits)
    SPD_CUDA_TRY(cudaMemcpyAsync(logits, lg, size_t(L.B) * m->cfg.vocab * sizeof(float), cudaMemcpyDeviceToHost, st));
  return SPD_OK;
}

extern "C" int spd_step_status(void* ws, const spd_model* m, const spd_prune_cfg* cfg, int n_seqs,
                               const int32_t* tiles_per_seq, const int32_t* text_len, void* stream) {
  StepLayout L;
  if (int rc = step_layout(m, cfg, n_seqs, tiles_per_seq, text_len, &L)) return rc;
  StepBufs s;
  step_carve(m, cfg, L, ws, &s);
  for (void* w : {static_cast<void*>(s.prune_ws), static_cast<void*>(s.proj_ws), static_cast<void*>(s.pre_ws)}) {
    if (w == s.proj_ws && !s.proj_bytes) continue;
    int v = 0;
    if (int rc = spd_workspace_status(w, stream, &v)) return rc;
    if (v) return v;
  }
  return SPD_OK;
}
