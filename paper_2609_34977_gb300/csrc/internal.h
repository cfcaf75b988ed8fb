// Internal declarations shared by the translation units of libspider.so.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include <utility>

#include "spider.h"

namespace spd {

// ---- errors ----------------------------------------------------------------------------------
int fail(int code, const char* fmt, ...);  // records the thread's message, returns code
#define SPD_CUDA_TRY(expr)                                                              \
  do {                                                                                  \
    cudaError_t e_ = (expr);                                                            \
    if (e_ != cudaSuccess)                                                              \
      return ::spd::fail(SPD_ECUDA, "%s failed: %s (%s:%d)", #expr, cudaGetErrorString(e_), \
                         __FILE__, __LINE__);                                           \
  } while (0)

// Clock budget of every bounded device-side wait (about half a second at 2 GHz).
constexpr long long kWaitBudget = 1ll << 30;

int num_sms();  // SM count of the current device


// Launches a kernel with programmatic stream serialization: it may be scheduled while the previous
// kernel of the stream is still running, and orders itself after it with griddepcontrol.wait.
//
// Rules every kernel of the library keeps under this overlap (the chain of launches in a stream
// can have several kernels resident at once, each waiting on its predecessor):
//  * before griddepcontrol.wait a kernel reads only data that no launch of the library writes
//    (weights, tensor maps, its own arguments) and writes nothing but its own shared memory;
//  * data that an earlier kernel of the stream wrote is read after the wait, and never through
//    the non-coherent path (no const __restrict__ pointers or ld.global.nc on it: PTX allows that
//    path only for data that stays unchanged while the kernel runs, and here the predecessor
//    writes it during this kernel's prologue);
//  * every kernel executes griddepcontrol.wait in at least one thread before it can complete, so
//    completion orders transitively: when kernel N passes its wait, every earlier kernel of the
//    stream has completed.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Bump allocator over a caller-provided workspace. The first 256 bytes hold the status word.
struct Carve {
  uint8_t* base;
  size_t used = 256;
  size_t cap;
  explicit Carve(void* b, size_t c) : base(static_cast<uint8_t*>(b)), cap(c) {}
  template <typename T>
  T* take(size_t n) {
    used = (used + 255) & ~size_t(255);
    T* p = reinterpret_cast<T*>(base ? base + used : nullptr);
    used += n * sizeof(T);
    return p;
  }
  bool fits() const { return used <= cap; }
  int* status() const { return reinterpret_cast<int*>(base); }
};

// ---- GEMM (tcgen05) --------------------------------------------------------------------------
enum Epi : int {
  EPI_F32 = SPD_EPI_F32,
  EPI_BF16 = SPD_EPI_BF16,
  EPI_BIAS_BF16 = SPD_EPI_BIAS_BF16,
  EPI_BIAS_GELU_BF16 = SPD_EPI_BIAS_GELU_BF16,
  EPI_ADD_F32 = SPD_EPI_ADD_F32,
  EPI_ROPE_BF16 = 16,  // rotary embedding on weight rows [0, rope_rows) laid out in rotary pairs
  EPI_SWIGLU_BF16 = 17, // SiLU(gate) * up from weight rows interleaved in gate/up half-warps
  EPI_QKV_BF16 = 18,    // rows [0, split): rotary, to out at row rows[t] (skipped when < 0);
                        // rows [split, n_out): to out2 at row t, rotary on the first rope_rows
  EPI_LSE_F32 = 19      // logit-lens statistics: for every group of 32 weight rows g and token t,
                        // float4 (m, s, u, 0) at out[t * ldo + g] with m = max z, s = sum e^(z - m),
                        // u = sum e^(z - m) (z - m) over the group's rows (rows past n_out left out)
};
// Number of 32-row groups of the logit-lens statistics of a V-word vocabulary.
__host__ __device__ inline int lse_groups(int V) { return (V + 31) / 32; }

struct GemmProblem {
  const CUtensorMap* map_w;  // weights [n_out][k] bf16, box 64 x 128 (optional)
  const void* w;             // the same weights (maps of other box heights are made from it)
  const void* x;             // activations [n_tok][k] bf16
  int n_out, n_tok, k;
  int epi;
  void* out;
  int ldo;
  const int32_t* rows;       // output row of token t (null = t)
  const uint16_t* bias;      // [n_out] bf16
  const int32_t* pos;        // rotary position of token t
  const void* rope;          // float2 [head_dim / 2]: freq_j = theta^(-2j / head_dim) as (hi, lo)
  int rope_rows, head_dim;
  int out_cols;              // valid output columns (SwiGLU: d_ffn)
  void* out2;                // EPI_QKV_BF16: second output, row stride ldo2, from weight row split
  const int32_t* rows2;      // EPI_QKV_BF16: row of token t in out2 (null = t)
  int ldo2, split;
  int n_tok_out;             // EPI_QKV_BF16: tokens whose first-output rows are stored (tracing)
  // Optional RMSNorm of the input, for the matrix-vector path only (gemm_fuses_norm): x is then
  // bf16(norm_gain * h[r] * rsqrt(mean h[r]^2 + norm_eps)) of fp32 rows r = norm_rows[t] (null = t)
  // of norm_h [.][k], and `x` is not read.
  const float* norm_h;
  const uint16_t* norm_gain;
  const int32_t* norm_rows;
  float norm_eps;
};
// True when gemm_run will run p on the matrix-vector path, which can apply the input RMSNorm itself.
bool gemm_fuses_norm(const GemmProblem& p);

// Scratch of stream-K partial slots (fp32, two per CTA) and per-tile arrival counters. The counters
// must be zero before a GEMM runs; every GEMM leaves them zero again when it completes.
constexpr size_t kGemmSlotFloats = size_t(10) << 20;
// Accumulation buffers of the data-parallel + remainder schedule: zero when a GEMM starts, left
// zero by every GEMM.
constexpr size_t kGemmAccFloats = size_t(4) << 20;
struct GemmScratch {
  float* partial;     // stream-K partial slots
  size_t partial_floats;
  float* acc;         // accumulation buffers (null: none)
  size_t acc_floats;
  int* counters;
  int n_counters;
  int* status;
};
// Clears the tile counters and the accumulation buffers of a workspace scratch on `stream` (done
// once per entry-point call, before its first GEMM).
int gemm_scratch_clear(const GemmScratch& s, cudaStream_t stream);
// Deterministic mode (process-wide): GEMMs sum every output element in a fixed order (split tiles
// through per-CTA partial slots summed in CTA order, residual updates as one read-modify-write per
// element) instead of fire-and-forget L2 reductions; repeated runs are then bit-identical.
int deterministic();
void set_deterministic(int on);

size_t gemm_scratch_bytes();                           // fixed-capacity scratch for any problem
int make_weight_map(CUtensorMap* map, const void* w, int n_out, int k);
// Tensor map of a dense bf16 matrix [outer][inner] (row stride inner elements) read in boxes of
// 64 columns x box_outer rows with the 128-byte swizzle; rows past `outer` read as zeros.
int make_operand_map(CUtensorMap* map, const void* ptr, int inner, int outer, int box_outer);

// ---- attention (tcgen05) ---------------------------------------------------------------------
// Causal attention of n_q active queries (q [n_q][n_heads * head_dim], rows grouped by sequence,
// positions ascending within a sequence) over the keys and values of their sequences (kv
// [n_kv][ldkv]: K of head g at column g * head_dim, V at v_off + g * head_dim). `tiles` (device
// int4 [n_tiles]): first query row, query count (1..128), first key row, sequence length.
int attention_run(const void* q, int n_q, const void* kv, int n_kv, int ldkv, int v_off, void* o,
                  int ldo, const int4* tiles, int n_tiles, const int32_t* q_pos, int n_heads,
                  int n_kv_heads, int head_dim, int* status, cudaStream_t stream, double ctx_sum);
constexpr int kAttnTileQ = 128;  // queries per attention tile
// The same attention when every tile holds ONE query at its sequence's last position (a decode
// step): tiles as above with query count 1; ctx_sum = the summed key counts.
int attention_decode_run(const void* q, const void* kv, int ldkv, int v_off, void* o, int ldo,
                         const int4* tiles, int n_tiles, int n_heads, int n_kv_heads, int head_dim,
                         cudaStream_t stream, double ctx_sum);
int gemm_run(const GemmProblem& p, const GemmScratch& s, cudaStream_t stream);

// ---- ASL-Skip online scores (Sec. 4.2.1, Eq. 6) -------------------------------------------------
// For candidate n (token cand[n], sequence seq_of[token]): E = entropy of softmax(logits[n]) / log V
// (mode kSkipEntropy, else 0; logits unread; with kSkipLse `logits` holds the float4 statistics of
// EPI_LSE_F32 instead, [n_cand][lse_groups(V)], merged here), F = (cos of h[token] to the mean h of its sequence's
// text tokens text[ts[b] .. ts[b+1]) (computed into tmean [B][D]) + 1) / 2 (mode kSkipItc, else 0),
// S_sa = ReLU(1 - E - F); s_skip[token] = (kSkipAccumulate ? s_skip[token] : 0) + w1 S_sa + add_slc;
// flag[n] = (s_skip[token] >= t_skip).
// kSkipDevice: the decision stays on the device: candidates with admit >= 0 are left alone, and
// one that reaches t_skip gets admit = layer, target = tgt (flag unused).
constexpr int kSkipEntropy = 1, kSkipItc = 2, kSkipAccumulate = 4, kSkipDevice = 8, kSkipLse = 16;
int skip_scores_run(const float* logits, int V, int n_cand, const float* h, int D, const int32_t* cand,
                    const int32_t* ts, const int32_t* text, const int32_t* seq_of, int B, float* tmean,
                    float w1, float add_slc, float t_skip, int mode, float* s_skip, uint8_t* flag,
                    cudaStream_t stream, int32_t* admit = nullptr, uint8_t* target = nullptr,
                    int layer = 0, int tgt = 0);
// Layer l's row lists built on the device from admission layers (see plan_lists_kernel).
constexpr int kPlanMaxSeqs = 1024;
int plan_lists_run(int T, int B, const int32_t* cu, const int32_t* pos, const int32_t* admit,
                   const uint8_t* target, int l, const int32_t* kv0, const int32_t* kvlen,
                   int32_t* arows, int32_t* amap, int32_t* apos, int32_t* frows, int4* tiles,
                   int max_tiles, cudaStream_t stream);

}  // namespace spd
