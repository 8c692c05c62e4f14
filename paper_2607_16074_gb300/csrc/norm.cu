// HBM-bound kernels of the backbone: the packer (gather into the canonical
// packed batch), RMSNorm, the final RMSNorm fused with the per-sample mean
// pool, and the RoPE (cos, sin) table.
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

// ---------------------------------------------------------------------------
// K1 packer.  One warp per packed token; 16-byte loads of the bf16 source
// row (a vision row or the text-embedding row of the token's id), widened to
// the fp32 residual stream.  The canonical packed batch is where the samples
// of all tenants are concatenated (§4.3); gather_src comes from the plan.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_pack(const int32_t* __restrict__ gather, int n_tokens,
                                              const uint16_t* __restrict__ vision, int64_t n_vision,
                                              const int32_t* __restrict__ text_ids, int64_t n_text,
                                              const uint16_t* __restrict__ table, int vocab, int d,
                                              float* __restrict__ x, int* status) {
    const int tok = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (tok >= n_tokens) return;
    const int src = gather[tok];
    const uint16_t* row = nullptr;
    if (src >= 0) {
        if (src < n_vision) row = vision + (size_t)src * d;
    } else {
        const int64_t p = -(int64_t)src - 1;
        if (p < n_text) {
            const int id = text_ids[p];
            if (id >= 0 && id < vocab) row = table + (size_t)id * d;
        }
    }
    if (row == nullptr && lane == 0) report(status, JNX_ERR_DEVICE_BOUNDS);
    float4* out = reinterpret_cast<float4*>(x + (size_t)tok * d);
    const int nchunk = d / 8;
    for (int c = lane; c < nchunk; c += 32) {
        float4 lo = make_float4(0.f, 0.f, 0.f, 0.f), hi = lo;
        if (row) {
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(row) + c);
            lo = make_float4(__uint_as_float(v.x << 16), __uint_as_float(v.x & 0xFFFF0000u),
                             __uint_as_float(v.y << 16), __uint_as_float(v.y & 0xFFFF0000u));
            hi = make_float4(__uint_as_float(v.z << 16), __uint_as_float(v.z & 0xFFFF0000u),
                             __uint_as_float(v.w << 16), __uint_as_float(v.w & 0xFFFF0000u));
        }
        out[2 * c] = lo;
        out[2 * c + 1] = hi;
    }
}

jnx_status pack_launch(const jnx_group* g, const uint16_t* vision, int64_t n_vision,
                       const int32_t* text_ids, int64_t n_text, const uint16_t* table, int vocab,
                       int d, float* x, int* status, cudaStream_t s) {
    if (d % 8) return fail(JNX_ERR_UNSUPPORTED, "pack: d %% 8 != 0");
    if (g->n_tokens == 0) return JNX_OK;
    k_pack<<<(g->n_tokens + 7) / 8, 256, 0, s>>>(g->gather_src, g->n_tokens, vision, n_vision,
                                                 text_ids, n_text, table, vocab, d, x, status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "pack: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// RMSNorm: one warp per row, the row held in registers (V float4 per lane),
// fp32 sum of squares reduced lane-wise then by a fixed shuffle tree, so a
// row's result does not depend on where it sits in the batch.
// ---------------------------------------------------------------------------
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <int V>
__global__ void __launch_bounds__(256) k_rmsnorm(const float* __restrict__ x,
                                                 const uint16_t* __restrict__ gamma, float eps,
                                                 int M, uint16_t* __restrict__ out) {
    constexpr int D = V * 128;
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= M) return;
    const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * D);
    float4 v[V];
    float ss = 0.f;
#pragma unroll
    for (int i = 0; i < V; ++i) {
        v[i] = __ldg(xr + lane + 32 * i);
        ss += v[i].x * v[i].x + v[i].y * v[i].y + v[i].z * v[i].z + v[i].w * v[i].w;
    }
    ss = warp_sum(ss);
    const float r = rsqrtf(ss / (float)D + eps);
    uint2* orow = reinterpret_cast<uint2*>(out + (size_t)row * D);
    const uint2* g2 = reinterpret_cast<const uint2*>(gamma);
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const uint2 gg = __ldg(g2 + lane + 32 * i);
        uint2 o;
        o.x = pack_bf2(v[i].x * r * bf2f(gg.x & 0xFFFF), v[i].y * r * bf2f(gg.x >> 16));
        o.y = pack_bf2(v[i].z * r * bf2f(gg.y & 0xFFFF), v[i].w * r * bf2f(gg.y >> 16));
        orow[lane + 32 * i] = o;
    }
}

// First half of a folded RMSNorm (the residual GEMM epilogue does the same for
// every later norm): y = bf16(x * gamma) and, per row and 256-column block,
// the sum of x^2; the consuming GEMM scales its output rows by
// rsqrt(sum / d + eps).  One warp per row.
template <int V>
__global__ void __launch_bounds__(256) k_rms_prep(const float* __restrict__ x,
                                                  const uint16_t* __restrict__ gamma, int M,
                                                  uint16_t* __restrict__ y, float* __restrict__ ss) {
    constexpr int D = V * 128;
    constexpr int P = D / 128;  // 128-column blocks: lane float4 i = b
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (row >= M) return;
    const float4* xr = reinterpret_cast<const float4*>(x + (size_t)row * D);
    float4 v[V];
#pragma unroll
    for (int i = 0; i < V; ++i) v[i] = __ldg(xr + lane + 32 * i);
#pragma unroll
    for (int b = 0; b < P; ++b) {
        float t = 0.f;
#pragma unroll
        t += v[b].x * v[b].x + v[b].y * v[b].y + v[b].z * v[b].z + v[b].w * v[b].w;
        t = warp_sum(t);
        if (lane == 0) ss[(size_t)row * P + b] = t;
    }
    uint2* orow = reinterpret_cast<uint2*>(y + (size_t)row * D);
    const uint2* g2 = reinterpret_cast<const uint2*>(gamma);
#pragma unroll
    for (int i = 0; i < V; ++i) {
        const uint2 gg = __ldg(g2 + lane + 32 * i);
        uint2 o;
        o.x = pack_bf2(v[i].x * bf2f(gg.x & 0xFFFF), v[i].y * bf2f(gg.x >> 16));
        o.y = pack_bf2(v[i].z * bf2f(gg.y & 0xFFFF), v[i].w * bf2f(gg.y >> 16));
        orow[lane + 32 * i] = o;
    }
}

jnx_status rms_prep_launch(const float* x, const uint16_t* gamma, int M, int d, uint16_t* y,
                           float* ss, cudaStream_t s) {
    if (M == 0) return JNX_OK;
    const int grid = (M + 7) / 8;
    switch (d) {
        case 256: k_rms_prep<2><<<grid, 256, 0, s>>>(x, gamma, M, y, ss); break;
        case 512: k_rms_prep<4><<<grid, 256, 0, s>>>(x, gamma, M, y, ss); break;
        case 1024: k_rms_prep<8><<<grid, 256, 0, s>>>(x, gamma, M, y, ss); break;
        case 2048: k_rms_prep<16><<<grid, 256, 0, s>>>(x, gamma, M, y, ss); break;
        case 4096: k_rms_prep<32><<<grid, 256, 0, s>>>(x, gamma, M, y, ss); break;
        default: return fail(JNX_ERR_UNSUPPORTED, "rms prep: d=%d not in {256..4096}", d);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "rms prep: %s", cudaGetErrorString(e));
}

jnx_status rmsnorm_launch(const float* x, const uint16_t* gamma, float eps, int M, int d,
                          uint16_t* out, cudaStream_t s) {
    if (M == 0) return JNX_OK;
    const int grid = (M + 7) / 8;
    switch (d) {
        case 256: k_rmsnorm<2><<<grid, 256, 0, s>>>(x, gamma, eps, M, out); break;
        case 512: k_rmsnorm<4><<<grid, 256, 0, s>>>(x, gamma, eps, M, out); break;
        case 1024: k_rmsnorm<8><<<grid, 256, 0, s>>>(x, gamma, eps, M, out); break;
        case 2048: k_rmsnorm<16><<<grid, 256, 0, s>>>(x, gamma, eps, M, out); break;
        case 4096: k_rmsnorm<32><<<grid, 256, 0, s>>>(x, gamma, eps, M, out); break;
        default: return fail(JNX_ERR_UNSUPPORTED, "rmsnorm: d=%d not in {256..4096}", d);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "rmsnorm: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// Final RMSNorm + mean pool.  One CTA per sample walks its rows in order
// (4 at a time); each thread owns columns tid, tid+256, ...; the row's sum
// of squares is reduced by a fixed tree.  pooled[s] = gamma * mean_t(x_t *
// rstd_t); hidden (optional) = bf16(x_t * rstd_t * gamma).
// ---------------------------------------------------------------------------
template <int C>  // columns per thread = d / 256
__global__ void __launch_bounds__(256) k_final_pool(const float* __restrict__ x,
                                                    const uint16_t* __restrict__ gamma, float eps,
                                                    const int* __restrict__ cu,
                                                    float* __restrict__ pooled,
                                                    uint16_t* __restrict__ hidden) {
    constexpr int D = C * 256;
    constexpr int R = 4;
    __shared__ float red[R][8];
    const int s = blockIdx.x;
    const int t0 = cu[s], t1 = cu[s + 1];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    float acc[C];
    float gm[C];
#pragma unroll
    for (int c = 0; c < C; ++c) {
        acc[c] = 0.f;
        gm[c] = bf2f(gamma[tid + 256 * c]);
    }
    for (int t = t0; t < t1; t += R) {
        float v[R][C];
        float ss[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            ss[r] = 0.f;
            const bool ok = t + r < t1;
#pragma unroll
            for (int c = 0; c < C; ++c) {
                v[r][c] = ok ? __ldg(x + (size_t)(t + r) * D + tid + 256 * c) : 0.f;
                ss[r] += v[r][c] * v[r][c];
            }
            ss[r] = warp_sum(ss[r]);
        }
        if (lane == 0) {
#pragma unroll
            for (int r = 0; r < R; ++r) red[r][warp] = ss[r];
        }
        __syncthreads();
        float rs[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            float tot = 0.f;
#pragma unroll
            for (int w = 0; w < 8; ++w) tot += red[r][w];
            rs[r] = rsqrtf(tot / (float)D + eps);
        }
        __syncthreads();
#pragma unroll
        for (int r = 0; r < R; ++r) {
            if (t + r >= t1) break;
#pragma unroll
            for (int c = 0; c < C; ++c) {
                const float y = v[r][c] * rs[r];
                acc[c] += y;
                if (hidden) hidden[(size_t)(t + r) * D + tid + 256 * c] = f2bf(y * gm[c]);
            }
        }
    }
    if (pooled) {
        const float inv = 1.0f / (float)(t1 - t0);
#pragma unroll
        for (int c = 0; c < C; ++c) pooled[(size_t)s * D + tid + 256 * c] = acc[c] * inv * gm[c];
    }
}

jnx_status final_pool_launch(const float* x, const uint16_t* gamma, float eps, const int* cu,
                             int S, int d, float* pooled, uint16_t* hidden, cudaStream_t s) {
    if (S == 0 || (!pooled && !hidden)) return JNX_OK;
    switch (d) {
        case 256: k_final_pool<1><<<S, 256, 0, s>>>(x, gamma, eps, cu, pooled, hidden); break;
        case 512: k_final_pool<2><<<S, 256, 0, s>>>(x, gamma, eps, cu, pooled, hidden); break;
        case 1024: k_final_pool<4><<<S, 256, 0, s>>>(x, gamma, eps, cu, pooled, hidden); break;
        case 2048: k_final_pool<8><<<S, 256, 0, s>>>(x, gamma, eps, cu, pooled, hidden); break;
        case 4096: k_final_pool<16><<<S, 256, 0, s>>>(x, gamma, eps, cu, pooled, hidden); break;
        default: return fail(JNX_ERR_UNSUPPORTED, "final_pool: d=%d not in {256..4096}", d);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "final_pool: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// RoPE table: (cos, sin) of pos * theta^(-2i/hd), evaluated in double and
// rounded to fp32 once.
// ---------------------------------------------------------------------------
// (cos, sin) of position p at frequency i, stored frequency-major
// (tab[i * max_pos + p]) so that rows of consecutive positions read
// consecutive entries.
__global__ void k_rope_table(float2* tab, int max_pos, int half, double theta) {
    const int idx = blockIdx.x * blockDim.x + threadIdx.x;
    if (idx >= max_pos * half) return;
    const int i = idx / max_pos, p = idx % max_pos;
    const double inv = pow(theta, -2.0 * (double)i / (double)(2 * half));
    double sn, cs;
    sincos((double)p * inv, &sn, &cs);
    tab[idx] = make_float2((float)cs, (float)sn);
}

jnx_status rope_table_launch(float2* tab, int max_pos, int hd, float theta, cudaStream_t s) {
    const int n = max_pos * (hd / 2);
    if (n == 0) return JNX_OK;
    k_rope_table<<<(n + 255) / 256, 256, 0, s>>>(tab, max_pos, hd / 2, (double)theta);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "rope table: %s", cudaGetErrorString(e));
}

}  // namespace jnx
