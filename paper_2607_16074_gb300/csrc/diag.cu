// Diagnostic entry points: two device routines that the hot-path kernels
// use, run on their own so that tests can pin them.  Neither is part of the
// grouped path.
//
//   jnx_diag_ex2_poly      the attention softmax's polynomial 2^x
//                          (ex2_poly2), evaluated on caller values
//   jnx_diag_bounded_wait  the bounded mbarrier wait every kernel's spins go
//                          through (mbar_wait), on a barrier that completes
//                          (arrive = 1) or that nothing ever arrives on
//                          (arrive = 0): the wait must give up after its
//                          limit and report JNX_ERR_TIMEOUT, never hang
#include "../../include/jnx_ops.h"
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {
namespace {

__global__ void k_diag_ex2(const float* __restrict__ x, float* __restrict__ y, int n) {
    const int i = 2 * (blockIdx.x * blockDim.x + threadIdx.x);
    if (i >= n) return;
    const bool two = i + 1 < n;
    float p0, p1;
    ex2_poly2(x[i], two ? x[i + 1] : 0.f, p0, p1);
    y[i] = p0;
    if (two) y[i + 1] = p1;
}

// One thread, one barrier in shared memory, no copy or MMA in flight.
__global__ void k_diag_wait(long long limit, int arrive, int* status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (arrive) mbar_arrive(&bar);  // completes phase 0
    if (!mbar_wait(&bar, 0, limit)) report(status, JNX_ERR_TIMEOUT);
}

}  // namespace
}  // namespace jnx

extern "C" jnx_status jnx_diag_ex2_poly(const float* x, float* y, int32_t n, void* stream) {
    jnx::clear_error();
    if (n < 0 || (n > 0 && (!x || !y)))
        return jnx::fail(JNX_ERR_INVALID_ARG, "diag ex2: null argument");
    if (n == 0) return JNX_OK;
    const int pairs = (n + 1) / 2;
    jnx::k_diag_ex2<<<(pairs + 255) / 256, 256, 0, static_cast<cudaStream_t>(stream)>>>(x, y, n);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : jnx::fail(JNX_ERR_CUDA, "diag ex2: %s", cudaGetErrorString(e));
}

extern "C" jnx_status jnx_diag_bounded_wait(int64_t limit_cycles, int32_t arrive,
                                            int32_t* status, void* stream) {
    jnx::clear_error();
    if (!status) return jnx::fail(JNX_ERR_INVALID_ARG, "diag wait: null status");
    // at most 2^31 SM clocks (about a second): a diagnostic, not a sleep
    if (limit_cycles <= 0 || limit_cycles > (1LL << 31))
        return jnx::fail(JNX_ERR_INVALID_ARG, "diag wait: limit %lld outside (0, 2^31]",
                         (long long)limit_cycles);
    jnx::k_diag_wait<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(limit_cycles, arrive ? 1 : 0,
                                                                      status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : jnx::fail(JNX_ERR_CUDA, "diag wait: %s", cudaGetErrorString(e));
}
