// Kernel-class tracing hooks (see trace.cu).
#pragma once
#include <cuda_runtime.h>

namespace spd {
enum TraceClass { TR_GEMM = 0, TR_ATTN = 1, TR_ROWS = 2, TR_PRUNE = 3 };
int trace_begin(cudaStream_t st);  // -1 when tracing is off or full
void trace_end(int slot, cudaStream_t st, int cls, double flops, double bytes);
// Device launch stamps: while stamping is on, the next launch of class cls records its start (the
// earliest CTA past its grid dependency wait) and end (the last CTA done) in globaltimer ns at the
// returned device address (two words); null when stamping is off or full.
unsigned long long* stamp_slot(int cls, double flops, double bytes);
}  // namespace spd
