// Tenant-private MLP action heads over the group's tenant segments.
//
// After the shared forward the features are split by the plan's slices and
// each tenant's own module runs on that tenant's samples only (App. A
// `split` / `decode`; §4.2 tenant-private loss and backward).  Samples are
// packed tenant by tenant, so group slot g owns packed samples
// [seg[g], seg[g+1]); every kernel takes a table of per-slot descriptors
// (weights and gradient buffers of that tenant) and walks the segments.
//
//   forward   z = p W1^T + b1, a = SiLU(z), y = a W2^T + b2
//   loss      l_t = sum (y - t)^2 / (n_t * width),  dy = 2 (y - t) / (n_t width)
//   backward  dW2 = dy^T a, db2 = sum dy, dz = (dy W2) * SiLU'(z),
//             dW1 = dz^T p, db1 = sum dz       -- into slot t only
// All sums run in a fixed order inside one thread or one CTA (no atomics),
// so a tenant's results are identical grouped or alone.
#include "jnx_dev.cuh"
#include "jnx_heads.h"

namespace jnx {

__device__ __forceinline__ float warp_sum_h(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float silu_f(float z) { return z / (1.0f + expf(-z)); }
__device__ __forceinline__ float silu_grad_f(float z) {
    const float s = 1.0f / (1.0f + expf(-z));
    return s * (1.0f + z * (1.0f - s));
}

// out[s, j] = sum_k in[s, k] W[j, k] + b[j] over the slot's samples; one warp
// per output column j, 8 samples at a time; lanes stride K in 8-element
// (16-byte) weight chunks.  LAYER 1 also stores a = SiLU(z); LAYER 2 scatters
// y to the caller's prediction buffer at each sample's target offset.
template <int LAYER>
__global__ void __launch_bounds__(256) k_mlp_fwd(const __grid_constant__ HeadTable tab, const float* __restrict__ in,
                                                 int ld_in, float* __restrict__ z_out,
                                                 float* __restrict__ a_out, int ld_out,
                                                 const int* __restrict__ sample_target,
                                                 float* __restrict__ preds) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int J = LAYER == 1 ? hs.d_hidden : hs.width;
    const int K = LAYER == 1 ? hs.d_in : hs.d_hidden;
    const uint16_t* W = LAYER == 1 ? hs.w1 : hs.w2;
    const uint16_t* B = LAYER == 1 ? hs.b1 : hs.b2;
    const int j = blockIdx.y * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= J) return;
    const uint4* wr = reinterpret_cast<const uint4*>(W + (size_t)j * K);
    const float bj = bf2f(B[j]);
    for (int s0 = hs.s0; s0 < hs.s1; s0 += 8) {
        const int ns = min(8, hs.s1 - s0);
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.f;
        for (int c = lane; c < K / 8; c += 32) {
            const uint4 w = __ldg(wr + c);
            const float wf[8] = {__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xFFFF0000u),
                                 __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xFFFF0000u),
                                 __uint_as_float(w.z << 16), __uint_as_float(w.z & 0xFFFF0000u),
                                 __uint_as_float(w.w << 16), __uint_as_float(w.w & 0xFFFF0000u)};
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                if (i < ns) {
                    const float4* xr =
                        reinterpret_cast<const float4*>(in + (size_t)(s0 + i) * ld_in + c * 8);
                    const float4 x0 = xr[0], x1 = xr[1];
                    acc[i] += x0.x * wf[0] + x0.y * wf[1] + x0.z * wf[2] + x0.w * wf[3] +
                              x1.x * wf[4] + x1.y * wf[5] + x1.z * wf[6] + x1.w * wf[7];
                }
            }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = warp_sum_h(acc[i]);
        if (lane < ns) {
            float v = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (i == lane) v = acc[i];
            const int s = s0 + lane;
            const float zz = v + bj;
            z_out[(size_t)s * ld_out + j] = zz;
            if (LAYER == 1) {
                a_out[(size_t)s * ld_out + j] = silu_f(zz);
            } else {
                preds[sample_target[s] + j] = zz;
            }
        }
    }
}

// Per-tenant loss and dy, one CTA per group slot, fixed-order reduction.
__global__ void __launch_bounds__(256) k_l2_loss(const __grid_constant__ HeadTable tab, const float* __restrict__ y,
                                                 int ld_y, const float* __restrict__ targets,
                                                 const int* __restrict__ sample_target,
                                                 float* __restrict__ dy, float* __restrict__ loss) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int W = hs.width;
    const int n = (hs.s1 - hs.s0) * W;
    const float inv = 1.0f / (float)n;
    float acc = 0.f;
    for (int i = threadIdx.x; i < n; i += 256) {
        const int s = hs.s0 + i / W, o = i % W;
        const float diff = y[(size_t)s * ld_y + o] - targets[sample_target[s] + o];
        acc += diff * diff;
        dy[(size_t)s * ld_y + o] = 2.0f * diff * inv;
    }
    __shared__ float red[8];
    acc = warp_sum_h(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < 8; ++w) t += red[w];
        loss[hs.tenant] = t * inv;
    }
}

// dW2[o, j] = sum_s dy[s, o] a[s, j]; db2[o] = sum_s dy[s, o].
__global__ void __launch_bounds__(256) k_mlp_dw2(const __grid_constant__ HeadTable tab, const float* __restrict__ dy,
                                                 const float* __restrict__ a, int ld) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int idx = blockIdx.y * 256 + threadIdx.x;
    if (idx >= hs.width * hs.d_hidden) return;
    const int o = idx / hs.d_hidden, j = idx % hs.d_hidden;
    float acc = 0.f, accb = 0.f;
    for (int s = hs.s0; s < hs.s1; ++s) {
        const float g = dy[(size_t)s * ld + o];
        acc += g * a[(size_t)s * ld + j];
        accb += g;
    }
    hs.g_w2[idx] = acc;
    if (j == 0) hs.g_b2[o] = accb;
}

// dz[s, j] = (sum_o dy[s, o] W2[o, j]) * SiLU'(z[s, j]); written over `a`.
__global__ void __launch_bounds__(256) k_mlp_dz(const __grid_constant__ HeadTable tab, const float* __restrict__ dy,
                                                const float* __restrict__ z,
                                                float* __restrict__ dz, int ld) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int j = blockIdx.y * 256 + threadIdx.x;
    if (j >= hs.d_hidden) return;
    for (int s = hs.s0; s < hs.s1; ++s) {
        float acc = 0.f;
        for (int o = 0; o < hs.width; ++o)
            acc += dy[(size_t)s * ld + o] * bf2f(hs.w2[(size_t)o * hs.d_hidden + j]);
        dz[(size_t)s * ld + j] = acc * silu_grad_f(z[(size_t)s * ld + j]);
    }
}

// dW1[j, k] = sum_s dz[s, j] p[s, k]; db1[j] = sum_s dz[s, j].  One CTA per
// (slot, j, 1024-column block); float4 columns.
__global__ void __launch_bounds__(256) k_mlp_dw1(const __grid_constant__ HeadTable tab, const float* __restrict__ dz,
                                                 int ld, const float* __restrict__ p, int ld_p) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int j = blockIdx.y;
    if (j >= hs.d_hidden) return;
    const int k4 = blockIdx.z * 256 + threadIdx.x;
    if (k4 * 4 < hs.d_in) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s = hs.s0; s < hs.s1; ++s) {
            const float g = dz[(size_t)s * ld + j];
            const float4 x = *reinterpret_cast<const float4*>(p + (size_t)s * ld_p + k4 * 4);
            acc.x += g * x.x;
            acc.y += g * x.y;
            acc.z += g * x.z;
            acc.w += g * x.w;
        }
        *reinterpret_cast<float4*>(hs.g_w1 + (size_t)j * hs.d_in + k4 * 4) = acc;
    }
    if (blockIdx.z == 0 && threadIdx.x == 0) {
        float accb = 0.f;
        for (int s = hs.s0; s < hs.s1; ++s) accb += dz[(size_t)s * ld + j];
        hs.g_b1[j] = accb;
    }
}

static jnx_status cuda_ok(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

jnx_status mlp_heads_forward(const HeadTable& tab, int n, int max_hidden, int max_width,
                             const float* pooled, int d, const int* sample_target,
                             const float* targets, float* preds, float* loss, HeadScratch ws,
                             cudaStream_t s) {
    if (n == 0) return JNX_OK;
    k_mlp_fwd<1><<<dim3(n, (max_hidden + 7) / 8), 256, 0, s>>>(tab, pooled, d, ws.z, ws.a, ws.ld,
                                                               sample_target, preds);
    k_mlp_fwd<2><<<dim3(n, (max_width + 7) / 8), 256, 0, s>>>(tab, ws.a, ws.ld, ws.y, nullptr,
                                                              ws.ld, sample_target, preds);
    k_l2_loss<<<n, 256, 0, s>>>(tab, ws.y, ws.ld, targets, sample_target, ws.dy, loss);
    return cuda_ok("mlp heads forward");
}

jnx_status mlp_heads_backward(const HeadTable& tab, int n, int max_hidden, int max_width,
                              int max_din, const float* pooled, int d, HeadScratch ws,
                              cudaStream_t s) {
    if (n == 0) return JNX_OK;
    k_mlp_dw2<<<dim3(n, (max_width * max_hidden + 255) / 256), 256, 0, s>>>(tab, ws.dy, ws.a,
                                                                             ws.ld);
    k_mlp_dz<<<dim3(n, (max_hidden + 255) / 256), 256, 0, s>>>(tab, ws.dy, ws.z, ws.dz, ws.ld);
    k_mlp_dw1<<<dim3(n, max_hidden, (max_din / 4 + 255) / 256), 256, 0, s>>>(tab, ws.dz, ws.ld,
                                                                              pooled, d);
    return cuda_ok("mlp heads backward");
}

}  // namespace jnx
