// jnx_op_gemm_rope_noalloc: the fused QKV projection + RoPE for callers that
// cannot allocate device memory.
//
// The ordinary entry point (jnx_op_gemm with JNX_EPI_ROPE) needs a caller
// workspace for its status word and its (cos, sin) table.  Some callers have
// no way to provide one: a plugin inside a serving process whose memory pool
// owns every device allocation, or a latency-critical batching worker that
// must not call cudaMalloc (it can synchronise the whole device) between
// requests.  They pass only inputs and outputs; the scratch lives in a
// file-scope __device__ array of fixed size that every GPU loading the
// library holds until the process exits.
//
// Rules of use:
//   - max_pos * head_dim / 2 must not exceed JNX_NOALLOC_MAX_ROPE_ENTRIES
//     (a 4 MiB table, plus 256 bytes of status word); larger requests are
//     rejected with JNX_ERR_UNSUPPORTED before anything is launched.
//   - The first call on a device looks up the array's device address with
//     cudaGetSymbolAddress (once per device, with that device current); make
//     that first call before any stream capture on that device.
//   - Every call on a device shares the one array.  Each call clears the
//     status word and rewrites the table rows it reads; calls that overlap
//     on the GPU (different streams, no ordering between them) race on it.
//   - A kernel-detected error (a position outside [0, max_pos): that row is
//     left unrotated; a wait that ran out of time) is recorded in the
//     array's status word; jnx_op_gemm_rope_noalloc_status reads and clears
//     it.
//   - Nothing here calls cudaMalloc, cudaFree or any allocating routine.
#include <mutex>

#include "../../include/jnx_ops.h"
#include "jnx_kernels.h"

namespace {

constexpr size_t kStatusBytes = 256;
constexpr size_t kTableEntries = JNX_NOALLOC_MAX_ROPE_ENTRIES;
constexpr size_t kScratchBytes = kStatusBytes + kTableEntries * sizeof(float2);

// The scratch itself.  In host code `g_scratch` is only a host-side stand-in
// for the symbol; its device address comes from cudaGetSymbolAddress.
static __device__ __align__(256) uint8_t g_scratch[kScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void* g_dev_addr[kMaxDevices] = {};

// Device address of g_scratch on the current device (looked up once).
jnx_status scratch_on_current_device(uint8_t** out) {
    int dev = -1;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess)
        return jnx::fail(JNX_ERR_CUDA, "gemm_rope_noalloc: cudaGetDevice: %s",
                         cudaGetErrorString(e));
    if (dev < 0 || dev >= kMaxDevices)
        return jnx::fail(JNX_ERR_UNSUPPORTED, "gemm_rope_noalloc: device %d >= %d", dev,
                         kMaxDevices);
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_dev_addr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_scratch);
        if (e != cudaSuccess || !p)
            return jnx::fail(JNX_ERR_CUDA, "gemm_rope_noalloc: cudaGetSymbolAddress: %s",
                             cudaGetErrorString(e));
        g_dev_addr[dev] = p;
    }
    *out = static_cast<uint8_t*>(g_dev_addr[dev]);
    return JNX_OK;
}

}  // namespace

extern "C" jnx_status jnx_op_gemm_rope_noalloc(const uint16_t* A, const uint16_t* W, int32_t M,
                                               int32_t N, int32_t K, uint16_t* out, int32_t ldo,
                                               const int32_t* pos, int32_t max_pos,
                                               int32_t rope_cols, int32_t head_dim,
                                               float rope_theta, void* stream) {
    jnx::clear_error();
    if (!A || !W || !out || !pos || M < 0)
        return jnx::fail(JNX_ERR_INVALID_ARG, "gemm_rope_noalloc: null argument");
    if (head_dim != 64 && head_dim != 128 && head_dim != 256)
        return jnx::fail(JNX_ERR_INVALID_ARG, "gemm_rope_noalloc: head_dim %d not in {64,128,256}",
                         head_dim);
    if (max_pos <= 0 || (size_t)max_pos * (size_t)(head_dim / 2) > kTableEntries)
        return jnx::fail(JNX_ERR_UNSUPPORTED,
                         "gemm_rope_noalloc: max_pos %d x head_dim/2 %d exceeds the fixed scratch "
                         "of %zu table entries",
                         max_pos, head_dim / 2, kTableEntries);
    if (rope_cols < 0 || rope_cols > N || rope_cols % head_dim)
        return jnx::fail(JNX_ERR_INVALID_ARG,
                         "gemm_rope_noalloc: rope_cols %d must be a multiple of head_dim %d "
                         "within N %d", rope_cols, head_dim, N);
    // the epilogue writes 16-byte vectors of whole rows
    if (ldo < N || ((size_t)ldo * 2) % 16 || reinterpret_cast<uintptr_t>(out) % 16)
        return jnx::fail(JNX_ERR_INVALID_ARG,
                         "gemm_rope_noalloc: out needs 16-byte aligned rows of >= %d", N);
    jnx_status st = jnx::gemm_check(M, N, K);
    if (st) return st;
    uint8_t* scratch = nullptr;
    if ((st = scratch_on_current_device(&scratch))) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemsetAsync(scratch, 0, kStatusBytes, s);  // status starts at zero
    if (e != cudaSuccess)
        return jnx::fail(JNX_ERR_CUDA, "gemm_rope_noalloc: %s", cudaGetErrorString(e));
    float2* table = reinterpret_cast<float2*>(scratch + kStatusBytes);
    if ((st = jnx::rope_table_launch(table, max_pos, head_dim, rope_theta, s))) return st;
    jnx::GemmParams p{};
    p.M = M;
    p.N = N;
    p.K = K;
    p.epi = jnx::EPI_ROPE;
    p.out = out;
    p.ldo = ldo;
    p.pos = pos;
    p.rope = table;
    p.rope_ld = max_pos;
    p.rope_cols = rope_cols;
    p.hd = head_dim;
    p.status = reinterpret_cast<int*>(scratch);
    return jnx::gemm_launch(A, K, W, K, p, s);
}

extern "C" jnx_status jnx_op_gemm_rope_noalloc_status(void* stream) {
    jnx::clear_error();
    uint8_t* scratch = nullptr;
    jnx_status st = scratch_on_current_device(&scratch);
    if (st) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int v = 0;
    // a copy into this pageable host int and a clear of the word: nothing
    // is allocated
    if (cudaMemcpyAsync(&v, scratch, sizeof v, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemsetAsync(scratch, 0, sizeof v, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return jnx::fail(JNX_ERR_CUDA, "gemm_rope_noalloc_status: %s",
                         cudaGetErrorString(cudaGetLastError()));
    if (v != 0) return jnx::fail(v, "a kernel reported status %d", v);
    return JNX_OK;
}
