// Kernel-class tracing: when enabled, every launch of the library is bracketed by a pair of CUDA
// events on its own stream, tagged with its class and its algorithmic work (flops and HBM bytes of
// the operation, not of the implementation). spd_trace_read sums device time and work per class.
#include <mutex>
#include <vector>

#include "internal.h"
#include "trace.h"

namespace spd {
namespace {

struct Trace {
  std::mutex mu;
  bool on = false;
  int cap = 0, used = 0;
  std::vector<cudaEvent_t> ev;
  std::vector<int> cls;
  std::vector<double> flops, bytes;
};
Trace& T() {
  static Trace t;
  return t;
}

// Device launch stamps: [start, end] globaltimer words per launch, written by the kernels.
struct Stamps {
  std::mutex mu;
  bool on = false;
  int cap = 0, used = 0;
  unsigned long long* dev = nullptr;
  std::vector<int> cls;
  std::vector<double> flops, bytes;
};
Stamps& S() {
  static Stamps s;
  return s;
}

}  // namespace

unsigned long long* stamp_slot(int cls, double flops, double bytes) {
  Stamps& s = S();
  if (!s.on) return nullptr;
  std::lock_guard<std::mutex> g(s.mu);
  if (s.used >= s.cap) return nullptr;
  const int k = s.used++;
  s.cls[k] = cls;
  s.flops[k] = flops;
  s.bytes[k] = bytes;
  return s.dev + 2 * size_t(k);
}

int trace_begin(cudaStream_t st) {
  Trace& t = T();
  if (!t.on) return -1;
  std::lock_guard<std::mutex> g(t.mu);
  if (t.used >= t.cap) return -1;
  const int s = t.used++;
  cudaEventRecord(t.ev[2 * s], st);
  return s;
}

void trace_end(int slot, cudaStream_t st, int cls, double flops, double bytes) {
  if (slot < 0) return;
  Trace& t = T();
  std::lock_guard<std::mutex> g(t.mu);
  cudaEventRecord(t.ev[2 * slot + 1], st);
  t.cls[slot] = cls;
  t.flops[slot] = flops;
  t.bytes[slot] = bytes;
}

}  // namespace spd

using namespace spd;

extern "C" int spd_trace_enable(int capacity) {
  Trace& t = T();
  std::lock_guard<std::mutex> g(t.mu);
  if (capacity <= 0) {
    t.on = false;
    return SPD_OK;
  }
  if (capacity > t.cap) {
    for (auto e : t.ev) cudaEventDestroy(e);
    t.ev.assign(2 * size_t(capacity), nullptr);
    for (auto& e : t.ev)
      if (cudaEventCreate(&e) != cudaSuccess) return fail(SPD_ECUDA, "cudaEventCreate failed");
    t.cap = capacity;
    t.cls.assign(capacity, 0);
    t.flops.assign(capacity, 0.0);
    t.bytes.assign(capacity, 0.0);
  }
  t.used = 0;
  t.on = true;
  return SPD_OK;
}

extern "C" int spd_trace_read(int cls, long long* launches, double* ms, double* flops, double* bytes) {
  Trace& t = T();
  std::lock_guard<std::mutex> g(t.mu);
  long long n = 0;
  double tot = 0.0, fl = 0.0, by = 0.0;
  for (int s = 0; s < t.used; ++s) {
    if (t.cls[s] != cls) continue;
    float e = 0.0f;
    if (cudaEventSynchronize(t.ev[2 * s + 1]) != cudaSuccess ||
        cudaEventElapsedTime(&e, t.ev[2 * s], t.ev[2 * s + 1]) != cudaSuccess)
      return fail(SPD_ECUDA, "trace event read failed");
    ++n;
    tot += e;
    fl += t.flops[s];
    by += t.bytes[s];
  }
  if (launches) *launches = n;
  if (ms) *ms = tot;
  if (flops) *flops = fl;
  if (bytes) *bytes = by;
  return SPD_OK;
}

// Launch stamps (see trace.h): every stamped launch writes the globaltimer ns of its first CTA past
// the grid dependency wait and of its last CTA's end. No event or other stream operation is added
// between launches, so the stamped step runs as it does unstamped.
extern "C" int spd_stamp_enable(int capacity) {
  Stamps& s = S();
  std::lock_guard<std::mutex> g(s.mu);
  if (capacity <= 0) {
    s.on = false;
    return SPD_OK;
  }
  if (capacity > s.cap) {
    if (s.dev) cudaFree(s.dev);
    s.dev = nullptr;
    if (cudaMalloc(&s.dev, 2 * sizeof(unsigned long long) * size_t(capacity)) != cudaSuccess)
      return fail(SPD_ECUDA, "cudaMalloc of the stamp buffer failed");
    s.cap = capacity;
    s.cls.assign(capacity, 0);
    s.flops.assign(capacity, 0.0);
    s.bytes.assign(capacity, 0.0);
  }
  std::vector<unsigned long long> init(2 * size_t(s.cap));
  for (size_t i = 0; i < init.size(); i += 2) {
    init[i] = ~0ull;  // start: atomicMin from the largest value
    init[i + 1] = 0;  // end: atomicMax from zero
  }
  SPD_CUDA_TRY(cudaDeviceSynchronize());
  SPD_CUDA_TRY(cudaMemcpy(s.dev, init.data(), init.size() * sizeof(unsigned long long),
                          cudaMemcpyHostToDevice));
  s.used = 0;
  s.on = true;
  return SPD_OK;
}

extern "C" int spd_stamp_read(int cls, long long* launches, double* ms, double* flops, double* bytes) {
  Stamps& s = S();
  std::lock_guard<std::mutex> g(s.mu);
  std::vector<unsigned long long> v(2 * size_t(s.used));
  SPD_CUDA_TRY(cudaDeviceSynchronize());
  if (s.used)
    SPD_CUDA_TRY(cudaMemcpy(v.data(), s.dev, v.size() * sizeof(unsigned long long),
                            cudaMemcpyDeviceToHost));
  long long n = 0;
  double tot = 0.0, fl = 0.0, by = 0.0;
  for (int k = 0; k < s.used; ++k) {
    if (s.cls[k] != cls || v[2 * k + 1] < v[2 * k]) continue;
    ++n;
    tot += double(v[2 * k + 1] - v[2 * k]) * 1e-6;
    fl += s.flops[k];
    by += s.bytes[k];
  }
  if (launches) *launches = n;
  if (ms) *ms = tot;
  if (flops) *flops = fl;
  if (bytes) *bytes = by;
  return SPD_OK;
}

extern "C" int spd_stamp_launch(int k, int* cls, unsigned long long* start_ns, unsigned long long* end_ns,
                                double* flops, double* bytes) {
  Stamps& s = S();
  std::lock_guard<std::mutex> g(s.mu);
  if (k < 0 || k >= s.used) return fail(SPD_EINVAL, "stamp %d not recorded (%d recorded)", k, s.used);
  unsigned long long v[2];
  SPD_CUDA_TRY(cudaDeviceSynchronize());
  SPD_CUDA_TRY(cudaMemcpy(v, s.dev + 2 * size_t(k), sizeof(v), cudaMemcpyDeviceToHost));
  if (cls) *cls = s.cls[k];
  if (start_ns) *start_ns = v[0];
  if (end_ns) *end_ns = v[1];
  if (flops) *flops = s.flops[k];
  if (bytes) *bytes = s.bytes[k];
  return SPD_OK;
}
