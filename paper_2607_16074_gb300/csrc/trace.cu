// Per-launch tracing: while enabled (on the calling host thread), every
// kernel the library launches is bracketed by two CUDA events on its stream,
// together with a kernel id and its algorithmic work (FLOPs for tensor-core
// kernels, HBM bytes for the others).  Off by default; when off, the hooks
// cost one thread-local load.
#include <vector>

#include "jnx_trace.h"

namespace jnx {

struct TraceState {
    bool on = false;
    int cap = 0;
    int count = 0;       // launches recorded
    int total = 0;       // launches seen (also counted past capacity)
    std::vector<cudaEvent_t> ev;
    std::vector<int> kind;
    std::vector<double> work;
};

static thread_local TraceState g_trace;

int trace_begin(int kind, double work, cudaStream_t s) {
    TraceState& t = g_trace;
    if (!t.on) return -1;
    ++t.total;
    if (t.count >= t.cap) return -1;
    const int i = t.count++;
    t.kind[i] = kind;
    t.work[i] = work;
    cudaEventRecord(t.ev[2 * i], s);
    return i;
}

void trace_end(int idx, cudaStream_t s) {
    if (idx < 0) return;
    cudaEventRecord(g_trace.ev[2 * idx + 1], s);
}

}  // namespace jnx

using namespace jnx;

extern "C" jnx_status jnx_trace_enable(int32_t capacity) {
    clear_error();
    TraceState& t = g_trace;
    if (capacity < 0) return fail(JNX_ERR_INVALID_ARG, "trace: negative capacity");
    if ((int)t.ev.size() < 2 * capacity) {
        for (int i = (int)t.ev.size(); i < 2 * capacity; ++i) {
            cudaEvent_t e;
            if (cudaEventCreate(&e) != cudaSuccess)
                return fail(JNX_ERR_CUDA, "trace: cudaEventCreate failed");
            t.ev.push_back(e);
        }
    }
    t.kind.assign(capacity, 0);
    t.work.assign(capacity, 0.0);
    t.cap = capacity;
    t.count = 0;
    t.total = 0;
    t.on = true;
    return JNX_OK;
}

extern "C" jnx_status jnx_trace_disable(void) {
    g_trace.on = false;
    return JNX_OK;
}

extern "C" int32_t jnx_trace_count(void) { return g_trace.total; }

extern "C" jnx_status jnx_trace_read(int32_t* kinds, float* ms, double* work, int32_t cap,
                                     int32_t* n_out) {
    clear_error();
    TraceState& t = g_trace;
    const int n = t.count < cap ? t.count : cap;
    for (int i = 0; i < n; ++i) {
        if (cudaEventSynchronize(t.ev[2 * i + 1]) != cudaSuccess)
            return fail(JNX_ERR_CUDA, "trace: event sync failed");
        float m = 0.f;
        if (cudaEventElapsedTime(&m, t.ev[2 * i], t.ev[2 * i + 1]) != cudaSuccess)
            return fail(JNX_ERR_CUDA, "trace: elapsed time failed");
        if (kinds) kinds[i] = t.kind[i];
        if (ms) ms[i] = m;
        if (work) work[i] = t.work[i];
    }
    if (n_out) *n_out = n;
    return JNX_OK;
}
