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

}  // namespace

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
