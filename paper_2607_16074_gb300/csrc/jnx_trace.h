// Internal tracing hooks (see trace.cu).
#pragma once
#include <cuda_runtime.h>

#include "jnx_host.h"

namespace jnx {

// Record the start event of a launch of `kind` doing `work` units; returns a
// handle for trace_end (or -1 when tracing is off or full).
int trace_begin(int kind, double work, cudaStream_t s);
void trace_end(int idx, cudaStream_t s);

// RAII bracket around one launch.
struct TraceScope {
    int idx;
    cudaStream_t s;
    TraceScope(int kind, double work, cudaStream_t st) : idx(trace_begin(kind, work, st)), s(st) {}
    ~TraceScope() { trace_end(idx, s); }
};

}  // namespace jnx
