// Tenant-private action heads over the group's tenant segments.
//
// After the shared forward the features are split by the plan's slices and
// each tenant's own module runs on that tenant's samples only (App. A
// `split` / `decode`; §5.2 tenant-private loss and backward).  Samples are
// packed tenant by tenant, so group slot g owns packed samples [s0, s1) and
// token rows [r0, r1); every kernel takes a table of per-slot descriptors
// (that tenant's weights and gradient buffers) and walks the segments.
//
// MLP head (on the pooled feature p):
//   z = p W1^T + b1, h = SiLU(z), y = h W2^T + b2
//   dW2 = dy^T h, db2 = sum dy, dz = (dy W2) * SiLU'(z), dW1 = dz^T p, db1 = sum dz
// Query head (on the sample's final normed rows X):
//   k = X Wk^T, v = X Wv^T            (tcgen05 GEMMs over the tenant's rows)
//   P = softmax(Q k^T / sqrt(dq)), O = P v, h = flatten(O), y = h Wout^T + bout
//   dWout = dy^T h, dbout = sum dy, dO = dy Wout,
//   dP = dO v^T, dS = P * (dP - rowsum(dP * P)), dv = P^T dO,
//   dk = dS^T Q / sqrt(dq), dQ = sum_s dS k / sqrt(dq), dWk = dk^T X, dWv = dv^T X
// Loss (both): l_t = sum (y - t)^2 / (n_t * width), dy = 2 (y - t) / (n_t width).
// All sums run in a fixed order inside one thread or one CTA (no atomics),
// so a tenant's results are identical whether it runs grouped or alone.
#include "jnx_dev.cuh"
#include "jnx_heads.h"
#include "jnx_kernels.h"

namespace jnx {

__device__ __forceinline__ float warp_sum_h(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max_h(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float silu_f(float z) { return z / (1.0f + expf(-z)); }
__device__ __forceinline__ float silu_grad_f(float z) {
    const float s = 1.0f / (1.0f + expf(-z));
    return s * (1.0f + z * (1.0f - s));
}

__device__ __forceinline__ void bf8_to_f(const uint4 w, float (&f)[8]) {
    f[0] = __uint_as_float(w.x << 16);
    f[1] = __uint_as_float(w.x & 0xFFFF0000u);
    f[2] = __uint_as_float(w.y << 16);
    f[3] = __uint_as_float(w.y & 0xFFFF0000u);
    f[4] = __uint_as_float(w.z << 16);
    f[5] = __uint_as_float(w.z & 0xFFFF0000u);
    f[6] = __uint_as_float(w.w << 16);
    f[7] = __uint_as_float(w.w & 0xFFFF0000u);
}

// ---------------------------------------------------------------------------
// Segmented linear layer: out[s, j] = sum_k in[s, k] W[j, k] + b[j] over the
// slot's samples.  One warp per output column j, 8 samples at a time; lanes
// stride K in 8-element (16-byte) weight chunks.
//   LAYER 1: MLP first layer (W1, b1; in = pooled); stores z and h = SiLU(z).
//   LAYER 2: output layer of either head (W2 or Wout; in = h); stores y and
//            scatters it to the caller's predictions at each target offset.
// ---------------------------------------------------------------------------
template <int LAYER>
__global__ void __launch_bounds__(256) k_head_lin(const __grid_constant__ HeadTable tab,
                                                  const float* __restrict__ in, int ld_in,
                                                  float* __restrict__ z_out, float* __restrict__ h_out,
                                                  int ld_out, const int* __restrict__ sample_target,
                                                  float* __restrict__ preds) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (LAYER == 1 && hs.kind != JNX_HEAD_MLP) return;
    const int J = LAYER == 1 ? hs.hid : hs.width;
    const int K = LAYER == 1 ? hs.d_in : hs.hid;
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
            float wf[8];
            bf8_to_f(__ldg(wr + c), wf);
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
            if (LAYER == 1)
                h_out[(size_t)s * ld_out + j] = silu_f(zz);
            else
                preds[sample_target[s] + j] = zz;
        }
    }
}

// Per-tenant loss and dy, one CTA per group slot, fixed-order reduction.
__global__ void __launch_bounds__(256) k_l2_loss(const __grid_constant__ HeadTable tab,
                                                 const float* __restrict__ y, int ld_y,
                                                 const float* __restrict__ targets,
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

// Output-layer weight gradient of either head: dW[o, j] = sum_s dy[s, o] h[s, j],
// db[o] = sum_s dy[s, o].
__global__ void __launch_bounds__(256) k_head_dw_out(const __grid_constant__ HeadTable tab,
                                                     const float* __restrict__ dy, int ld_y,
                                                     const float* __restrict__ h, int ld_h) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int idx = blockIdx.y * 256 + threadIdx.x;
    if (idx >= hs.width * hs.hid) return;
    const int o = idx / hs.hid, j = idx % hs.hid;
    float acc = 0.f, accb = 0.f;
    for (int s = hs.s0; s < hs.s1; ++s) {
        const float g = dy[(size_t)s * ld_y + o];
        acc += g * h[(size_t)s * ld_h + j];
        accb += g;
    }
    hs.g_w2[idx] = hs.accum ? hs.g_w2[idx] + acc : acc;
    if (j == 0) hs.g_b2[o] = hs.accum ? hs.g_b2[o] + accb : accb;
}

// Gradient into the output layer's input: dh[s, j] = (sum_o dy[s, o] W[o, j])
// times SiLU'(z[s, j]) for an MLP slot (dz), plain for a query head (dO).
// One thread per column j, 8 samples at a time so W is read once per 8.
__global__ void __launch_bounds__(256) k_head_back_in(const __grid_constant__ HeadTable tab,
                                                      const float* __restrict__ dy, int ld_y,
                                                      const float* __restrict__ z, int ld_h,
                                                      float* __restrict__ dh) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int j = blockIdx.y * 256 + threadIdx.x;
    if (j >= hs.hid) return;
    for (int s0 = hs.s0; s0 < hs.s1; s0 += 8) {
        const int ns = min(8, hs.s1 - s0);
        float acc[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) acc[i] = 0.f;
        for (int o = 0; o < hs.width; ++o) {
            const float w = bf2f(hs.w2[(size_t)o * hs.hid + j]);
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (i < ns) acc[i] += dy[(size_t)(s0 + i) * ld_y + o] * w;
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            if (i >= ns) break;
            const size_t at = (size_t)(s0 + i) * ld_h + j;
            dh[at] = hs.kind == JNX_HEAD_MLP ? acc[i] * silu_grad_f(z[at]) : acc[i];
        }
    }
}

// MLP first-layer gradient: dW1[j, k] = sum_s dz[s, j] p[s, k]; db1[j] = sum_s dz[s, j].
// One CTA per (slot, j, 1024-column block); float4 columns.
__global__ void __launch_bounds__(256) k_mlp_dw1(const __grid_constant__ HeadTable tab,
                                                 const float* __restrict__ dz, int ld,
                                                 const float* __restrict__ p, int ld_p) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_MLP) return;
    const int j = blockIdx.y;
    if (j >= hs.hid) return;
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
        float4* dst = reinterpret_cast<float4*>(hs.g_w1 + (size_t)j * hs.d_in + k4 * 4);
        if (hs.accum) {
            const float4 old = *dst;
            acc.x += old.x;
            acc.y += old.y;
            acc.z += old.z;
            acc.w += old.w;
        }
        *dst = acc;
    }
    if (blockIdx.z == 0 && threadIdx.x == 0) {
        float accb = 0.f;
        for (int s = hs.s0; s < hs.s1; ++s) accb += dz[(size_t)s * ld + j];
        hs.g_b1[j] = hs.accum ? hs.g_b1[j] + accb : accb;
    }
}

// ---------------------------------------------------------------------------
// Query head, per sample.  One CTA per packed sample of a query-head slot;
// the tenant's learned queries (nq <= 32 of width dq) sit in shared memory.
// P (normalised attention) for sample s is stored key-major at P + nq * cu[s]:
// element (query q, key j) at j * nq + q (nq a multiple of 4).
// ---------------------------------------------------------------------------
constexpr int kMaxQ = 32;

__global__ void __launch_bounds__(256, 1) k_xattn_fwd(const __grid_constant__ HeadTable tab, int g0,
                                                   const int* __restrict__ cu,
                                                   const int* __restrict__ sample_slot,
                                                   int sample0, const float* __restrict__ kbuf,
                                                   const float* __restrict__ vbuf, int ldkv,
                                                   float* __restrict__ P, float* __restrict__ h,
                                                   int ld_h) {
    extern __shared__ float xs[];  // Q [nq][dq]
    const int s = sample0 + blockIdx.x;
    const HeadSlot& hs = tab.slot[sample_slot[s] - g0];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, dq = hs.dq;
    const int r0 = cu[s], L = cu[s + 1] - r0;
    const float scale = rsqrtf((float)dq);
    for (int i = threadIdx.x; i < nq * dq; i += 256) xs[i] = bf2f(hs.q[i]);
    __syncthreads();
    float* Ps = P + (size_t)nq * r0;
    // scores: one thread per key, all queries
    for (int j = threadIdx.x; j < L; j += 256) {
        float acc[kMaxQ];
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q) acc[q] = 0.f;
        const float4* kr = reinterpret_cast<const float4*>(kbuf + (size_t)(r0 + j) * ldkv);
        for (int c4 = 0; c4 < dq / 4; ++c4) {
            const float4 kv = kr[c4];
#pragma unroll
            for (int q = 0; q < kMaxQ; ++q) {
                if (q < nq) {
                    const float* qq = xs + q * dq + 4 * c4;
                    acc[q] += qq[0] * kv.x + qq[1] * kv.y + qq[2] * kv.z + qq[3] * kv.w;
                }
            }
        }
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q)
            if (q < nq) Ps[(size_t)j * nq + q] = acc[q] * scale;
    }
    __syncthreads();
    // softmax per query (key-major storage: element (q, j) at j * nq + q);
    // one warp per query
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int q = warp; q < nq; q += 8) {
        float m = -INFINITY;
        for (int j = lane; j < L; j += 32) m = fmaxf(m, Ps[(size_t)j * nq + q]);
        m = warp_max_h(m);
        float sum = 0.f;
        for (int j = lane; j < L; j += 32) {
            const float e = expf(Ps[(size_t)j * nq + q] - m);
            Ps[(size_t)j * nq + q] = e;
            sum += e;
        }
        sum = warp_sum_h(sum);
        const float inv = 1.0f / sum;
        for (int j = lane; j < L; j += 32) Ps[(size_t)j * nq + q] *= inv;
    }
    __syncthreads();
    // O = P v: one thread per value column c
    for (int c = threadIdx.x; c < dq; c += 256) {
        float acc[kMaxQ];
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q) acc[q] = 0.f;
        for (int j = 0; j < L; ++j) {
            const float vv = vbuf[(size_t)(r0 + j) * ldkv + c];
            const float4* pj = reinterpret_cast<const float4*>(Ps + (size_t)j * nq);
#pragma unroll
            for (int q4 = 0; q4 < kMaxQ / 4; ++q4) {
                if (4 * q4 < nq) {
                    const float4 pp = pj[q4];
                    acc[4 * q4 + 0] += pp.x * vv;
                    acc[4 * q4 + 1] += pp.y * vv;
                    acc[4 * q4 + 2] += pp.z * vv;
                    acc[4 * q4 + 3] += pp.w * vv;
                }
            }
        }
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q)
            if (q < nq) h[(size_t)s * ld_h + q * dq + c] = acc[q];
    }
}

// Backward per sample: dP, dS (stored over dPbuf), dv, dk rows, and this
// sample's dQ contribution (summed per tenant later in sample order).
__global__ void __launch_bounds__(256, 1) k_xattn_bwd(const __grid_constant__ HeadTable tab, int g0,
                                                   const int* __restrict__ cu,
                                                   const int* __restrict__ sample_slot,
                                                   int sample0, const float* __restrict__ kbuf,
                                                   const float* __restrict__ vbuf, int ldkv,
                                                   const float* __restrict__ P,
                                                   float* __restrict__ dS,
                                                   const float* __restrict__ dO, int ld_h,
                                                   float* __restrict__ dk, float* __restrict__ dv,
                                                   float* __restrict__ dQs) {
    extern __shared__ float xs[];  // Q [nq][dq], then dO [nq][dq]
    const int s = sample0 + blockIdx.x;
    const HeadSlot& hs = tab.slot[sample_slot[s] - g0];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, dq = hs.dq;
    const int r0 = cu[s], L = cu[s + 1] - r0;
    const float scale = rsqrtf((float)dq);
    float* Qs = xs;
    float* dOs = xs + nq * dq;
    for (int i = threadIdx.x; i < nq * dq; i += 256) {
        Qs[i] = bf2f(hs.q[i]);
        dOs[i] = dO[(size_t)s * ld_h + i];
    }
    __syncthreads();
    const float* Ps = P + (size_t)nq * r0;
    float* dSs = dS + (size_t)nq * r0;
    // dP[q, j] = dO[q, :] . v[j, :]
    for (int j = threadIdx.x; j < L; j += 256) {
        float acc[kMaxQ];
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q) acc[q] = 0.f;
        const float4* vr = reinterpret_cast<const float4*>(vbuf + (size_t)(r0 + j) * ldkv);
        for (int c4 = 0; c4 < dq / 4; ++c4) {
            const float4 vv = vr[c4];
#pragma unroll
            for (int q = 0; q < kMaxQ; ++q) {
                if (q < nq) {
                    const float* o = dOs + q * dq + 4 * c4;
                    acc[q] += o[0] * vv.x + o[1] * vv.y + o[2] * vv.z + o[3] * vv.w;
                }
            }
        }
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q)
            if (q < nq) dSs[(size_t)j * nq + q] = acc[q];
    }
    __syncthreads();
    // dS = P * (dP - sum_j dP * P), one warp per query (key-major storage)
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int q = warp; q < nq; q += 8) {
        float t = 0.f;
        for (int j = lane; j < L; j += 32) t += dSs[(size_t)j * nq + q] * Ps[(size_t)j * nq + q];
        t = warp_sum_h(t);
        for (int j = lane; j < L; j += 32) {
            const size_t at = (size_t)j * nq + q;
            dSs[at] = Ps[at] * (dSs[at] - t);
        }
    }
    __syncthreads();
    // per value column c: dv[j, c], dk[j, c] for every key j, and dQ[:, c]
    for (int c = threadIdx.x; c < dq; c += 256) {
        float dq_acc[kMaxQ];
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q) dq_acc[q] = 0.f;
        for (int j = 0; j < L; ++j) {
            float a_v = 0.f, a_k = 0.f;
            const float kk = kbuf[(size_t)(r0 + j) * ldkv + c];
            const float4* pj = reinterpret_cast<const float4*>(Ps + (size_t)j * nq);
            const float4* dj = reinterpret_cast<const float4*>(dSs + (size_t)j * nq);
#pragma unroll
            for (int q4 = 0; q4 < kMaxQ / 4; ++q4) {
                if (4 * q4 < nq) {
                    const float4 p4 = pj[q4], d4 = dj[q4];
                    const float pp[4] = {p4.x, p4.y, p4.z, p4.w};
                    const float dd[4] = {d4.x, d4.y, d4.z, d4.w};
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int q = 4 * q4 + e;
                        a_v += pp[e] * dOs[q * dq + c];
                        a_k += dd[e] * Qs[q * dq + c];
                        dq_acc[q] += dd[e] * kk;
                    }
                }
            }
            dv[(size_t)(r0 + j) * ldkv + c] = a_v;
            dk[(size_t)(r0 + j) * ldkv + c] = a_k * scale;
        }
#pragma unroll
        for (int q = 0; q < kMaxQ; ++q)
            if (q < nq) dQs[(size_t)s * ld_h + q * dq + c] = dq_acc[q] * scale;
    }
}

// dQ_t = sum over the slot's samples (in order) of their contributions.
__global__ void __launch_bounds__(256) k_xattn_dq(const __grid_constant__ HeadTable tab,
                                                  const float* __restrict__ dQs, int ld_h) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int i = blockIdx.y * 256 + threadIdx.x;
    if (i >= hs.nq * hs.dq) return;
    float acc = 0.f;
    for (int s = hs.s0; s < hs.s1; ++s) acc += dQs[(size_t)s * ld_h + i];
    hs.g_q[i] = hs.accum ? hs.g_q[i] + acc : acc;
}

// dW[c, e] = sum over the slot's token rows r of g[r, c] * X[r, e], for
// g = dk (-> dWk) and g = dv (-> dWv): a GEMM whose reduction runs over the
// tenant's rows, on bf16 mma.sync (m16n8k16) with fp32 accumulation.  One
// CTA per 64 x 128 output tile, 4 warps in a 2 x 2 layout (32 x 64 each);
// rows stream through shared memory in chunks of 32.  The fp32 g is split
// while staged into g_hi = bf16(g) and g_lo = bf16(g - g_hi) and both are
// multiplied (X is exact in bf16), which keeps the result at fp32 accuracy;
// both operands are row-major in r (MN-major) and are read with
// ldmatrix.trans; X arrives by cp.async.  Fixed reduction order.
namespace wg {
constexpr int BMC = 64, BNE = 128, BR = 32;
}

__global__ void __launch_bounds__(128) k_xattn_wgrad(const __grid_constant__ HeadTable tab,
                                                     const float* __restrict__ dk,
                                                     const float* __restrict__ dv, int ldkv,
                                                     const uint16_t* __restrict__ X, int ldx) {
    using namespace wg;
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int which = blockIdx.z & 1;
    const int c0 = blockIdx.y * BMC;            // dq rows of the tile
    const int e0 = (blockIdx.z >> 1) * BNE;     // d columns of the tile
    if (c0 >= hs.dq || e0 >= hs.d_in) return;
    const float* G = which ? dv : dk;
    float* out = which ? hs.g_wv : hs.g_wk;
    __shared__ __align__(128) uint8_t sA[2][2][BR * BMC * 2];  // [buf][hi/lo][r][c] bf16
    __shared__ __align__(128) uint8_t sB[2][BR * BNE * 2];  // [r][e] bf16, 256-byte rows
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wm = warp & 1, wn = warp >> 1;
    const uint32_t aA = smem_u32(sA), aB = smem_u32(sB);
    // row r, 16-byte chunk ch of a tile with `cpr` chunks per row, XOR-swizzled
    auto swz = [](int r, int ch, int cpr) { return (uint32_t)(r * cpr * 16 + ((ch ^ (r & 7)) << 4)); };

    float acc[2][8][4];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j][0] = acc[i][j][1] = acc[i][j][2] = acc[i][j][3] = 0.f;

    // A staging: thread -> (row = tid / 4, 16 consecutive c at (tid % 4) * 16)
    const int ar = tid >> 2, ac = (tid & 3) * 16;
    float4 areg[4];
    auto load_a = [&](int r) {
        const bool ok = r + ar < hs.r1;
        const float4* src = reinterpret_cast<const float4*>(G + (size_t)(r + ar) * ldkv + c0 + ac);
#pragma unroll
        for (int i = 0; i < 4; ++i) areg[i] = ok ? src[i] : make_float4(0.f, 0.f, 0.f, 0.f);
    };
    auto store_a = [&](int buf) {
        uint8_t* hi_base = sA[buf][0];
        uint8_t* lo_base = sA[buf][1];
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const float v[8] = {areg[2 * h].x,     areg[2 * h].y,     areg[2 * h].z,
                                areg[2 * h].w,     areg[2 * h + 1].x, areg[2 * h + 1].y,
                                areg[2 * h + 1].z, areg[2 * h + 1].w};
            uint32_t hw[4], lw[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                hw[q] = pack_bf2(v[2 * q], v[2 * q + 1]);
                const float h0 = __uint_as_float(hw[q] << 16);
                const float h1 = __uint_as_float(hw[q] & 0xFFFF0000u);
                lw[q] = pack_bf2(v[2 * q] - h0, v[2 * q + 1] - h1);
            }
            const uint32_t off = swz(ar, ac / 8 + h, BMC / 8);
            *reinterpret_cast<uint4*>(hi_base + off) = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            *reinterpret_cast<uint4*>(lo_base + off) = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
    };
    auto load_b = [&](int r, int buf) {
        for (int i = tid; i < BR * (BNE / 8); i += 128) {
            const int rr = i / (BNE / 8), ch = i % (BNE / 8);
            const bool ok = r + rr < hs.r1;
            cp_async16(aB + buf * BR * BNE * 2 + swz(rr, ch, BNE / 8),
                       ok ? (const void*)(X + (size_t)(r + rr) * ldx + e0 + ch * 8)
                          : (const void*)X,
                       ok);
        }
    };

    const int mi = lane >> 3, rr8 = lane & 7;
    int buf = 0;
    if (hs.r0 < hs.r1) {
        load_a(hs.r0);
        load_b(hs.r0, 0);
        cp_async_commit();
        store_a(0);
    }
    for (int r = hs.r0; r < hs.r1; r += BR) {
        const bool more = r + BR < hs.r1;
        if (more) {
            load_a(r + BR);
            load_b(r + BR, buf ^ 1);
        }
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t a_base = aA + buf * 2 * BR * BMC * 2, b_base = aB + buf * BR * BNE * 2;
#pragma unroll
        for (int ks = 0; ks < BR / 16; ++ks) {
            uint32_t af[2][2][4];  // [hi/lo][m-tile][regs]
#pragma unroll
            for (int part = 0; part < 2; ++part)
#pragma unroll
                for (int im = 0; im < 2; ++im) {
                    // matrices (m 0-7, k 0-7), (m 8-15, k 0-7), (m 0-7, k 8-15), (m 8-15, k 8-15)
                    const int kr = ks * 16 + rr8 + 8 * (mi >> 1);
                    const int mch = (wm * 32 + im * 16) / 8 + (mi & 1);
                    ldsm_x4_t(a_base + part * BR * BMC * 2 + swz(kr, mch, BMC / 8),
                              af[part][im][0], af[part][im][1], af[part][im][2], af[part][im][3]);
                }
#pragma unroll
            for (int np = 0; np < 4; ++np) {
                // matrices (k 0-7, n 0-7), (k 8-15, n 0-7), (k 0-7, n 8-15), (k 8-15, n 8-15)
                const int kr = ks * 16 + rr8 + 8 * (mi & 1);
                const int nch = (wn * 64 + np * 16) / 8 + (mi >> 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(b_base + swz(kr, nch, BNE / 8), b0, b1, b2, b3);
#pragma unroll
                for (int part = 0; part < 2; ++part)
#pragma unroll
                    for (int im = 0; im < 2; ++im) {
                        const uint32_t* a = af[part][im];
                        mma_bf16(acc[im][2 * np], a[0], a[1], a[2], a[3], b0, b1);
                        mma_bf16(acc[im][2 * np + 1], a[0], a[1], a[2], a[3], b2, b3);
                    }
            }
        }
        __syncthreads();
        if (more) store_a(buf ^ 1);
        buf ^= 1;
    }
    const int g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int im = 0; im < 2; ++im) {
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int c = c0 + wm * 32 + im * 16 + g;
            const int e = e0 + wn * 64 + j * 8 + 2 * t;
            float2* d0 = reinterpret_cast<float2*>(out + (size_t)c * hs.d_in + e);
            float2* d1 = reinterpret_cast<float2*>(out + (size_t)(c + 8) * hs.d_in + e);
            float2 v0 = make_float2(acc[im][j][0], acc[im][j][1]);
            float2 v1 = make_float2(acc[im][j][2], acc[im][j][3]);
            if (hs.accum) {
                const float2 o0 = *d0, o1 = *d1;
                v0.x += o0.x;
                v0.y += o0.y;
                v1.x += o1.x;
                v1.y += o1.y;
            }
            *d0 = v0;
            *d1 = v1;
        }
    }
}

// ---------------------------------------------------------------------------
// launchers
// ---------------------------------------------------------------------------
static jnx_status cuda_ok(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

jnx_status heads_forward_launch(const HeadTable& tab, const HeadBatch& b, const HeadScratch& ws,
                                const float* pooled, int d, const int* cu, const int* sample_slot,
                                const int* sample_target, const float* targets, float* preds,
                                float* loss, cudaStream_t s) {
    if (b.n == 0) return JNX_OK;
    if (b.any_mlp)
        k_head_lin<1><<<dim3(b.n, (b.max_hid + 7) / 8), 256, 0, s>>>(
            tab, pooled, d, ws.z, ws.h, ws.ld_h, sample_target, preds);
    if (b.any_xattn) {
        const size_t smem = (size_t)b.max_nq * b.max_dq * sizeof(float);
        k_xattn_fwd<<<b.sample1 - b.sample0, 256, smem, s>>>(tab, b.g0, cu, sample_slot,
                                                             b.sample0, ws.kbuf, ws.vbuf, ws.ldkv,
                                                             ws.P, ws.h, ws.ld_h);
    }
    k_head_lin<2><<<dim3(b.n, (b.max_width + 7) / 8), 256, 0, s>>>(tab, ws.h, ws.ld_h, ws.y,
                                                                   nullptr, ws.ld_y,
                                                                   sample_target, preds);
    if (targets)  // without targets (inference) there is no loss
        k_l2_loss<<<b.n, 256, 0, s>>>(tab, ws.y, ws.ld_y, targets, sample_target, ws.dy, loss);
    return cuda_ok("heads forward");
}

jnx_status heads_backward_launch(const HeadTable& tab, const HeadBatch& b, const HeadScratch& ws,
                                 const float* pooled, int d, const uint16_t* hidden,
                                 const int* cu, const int* sample_slot, cudaStream_t s) {
    if (b.n == 0) return JNX_OK;
    k_head_dw_out<<<dim3(b.n, (b.max_width * b.max_hid + 255) / 256), 256, 0, s>>>(
        tab, ws.dy, ws.ld_y, ws.h, ws.ld_h);
    k_head_back_in<<<dim3(b.n, (b.max_hid + 255) / 256), 256, 0, s>>>(tab, ws.dy, ws.ld_y, ws.z,
                                                                      ws.ld_h, ws.dh);
    if (b.any_mlp)
        k_mlp_dw1<<<dim3(b.n, b.max_mlp_hid, (d / 4 + 255) / 256), 256, 0, s>>>(tab, ws.dh,
                                                                               ws.ld_h, pooled, d);
    if (b.any_xattn) {
        const size_t smem = 2 * (size_t)b.max_nq * b.max_dq * sizeof(float);
        k_xattn_bwd<<<b.sample1 - b.sample0, 256, smem, s>>>(
            tab, b.g0, cu, sample_slot, b.sample0, ws.kbuf, ws.vbuf, ws.ldkv, ws.P, ws.dS, ws.dh,
            ws.ld_h, ws.dk, ws.dv, ws.dQs);
        k_xattn_dq<<<dim3(b.n, (b.max_nq * b.max_dq + 255) / 256), 256, 0, s>>>(tab, ws.dQs,
                                                                                 ws.ld_h);
        k_xattn_wgrad<<<dim3(b.n, b.max_dq / wg::BMC, 2 * (d / wg::BNE)), 128, 0, s>>>(
            tab, ws.dk, ws.dv, ws.ldkv, hidden, d);
    }
    return cuda_ok("heads backward");
}

jnx_status heads_set_smem() {
    static std::atomic<uint64_t> fwd{0}, bwd{0};
    const int mx = 2 * kMaxQ * 512 * (int)sizeof(float);
    if (set_smem_limit(reinterpret_cast<const void*>(k_xattn_fwd), mx, fwd) != cudaSuccess ||
        set_smem_limit(reinterpret_cast<const void*>(k_xattn_bwd), mx, bwd) != cudaSuccess)
        return cuda_ok("heads smem attribute");
    return JNX_OK;
}

}  // namespace jnx
