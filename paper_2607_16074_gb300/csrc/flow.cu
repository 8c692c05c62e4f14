// Flow-matching action expert (a DiT head) as the tenant-private module
// (§3.1: a diffusion / flow-matching action expert can be the action module;
// §5.2: QwenGR00T's GR00T-style flow-matching head, the tenant-private part
// over the shared VLM).  The expert's equations are in jnx.h.
//
// Rows: the group's action tokens, r = s C + c for packed sample s and chunk
// step c (M_a = S C rows, a tenant's rows contiguous like its samples), and
// the backbone's token rows for the context.  Every per-tenant projection
// is one segmented tcgen05 GEMM over the group (gemm_launch_seg: a tenant's
// rows times its slice of the stacked weights); weight gradients are
// k_seg_wgrad (mma.sync, a tenant's rows in a fixed order); the attention
// (C <= 64 queries per sample against its L context rows and C action rows)
// and the small per-row / per-sample pieces run on CUDA cores in fp32.
#include <algorithm>
#include <cmath>
#include <vector>

#include "../../include/jnx.h"
#include "jnx_bwd.h"
#include "jnx_dev.cuh"
#include "jnx_kernels.h"
#include "jnx_trace.h"

namespace jnx {
namespace {

constexpr int kHd = 64;       // attention head width
constexpr int kMaxC = 64;     // longest action chunk
constexpr int kMaxD = 64;     // widest action
constexpr float kEps = 1e-6f;
constexpr float kLog2e = 1.4426950408889634f;

// Per-slot view of the group: tenant and packed samples [s0, s1).
struct FlowSlots {
    int n;
    int tenant[kSegMaxSlots];
    int s0[kSegMaxSlots], s1[kSegMaxSlots];
};

struct FlowDims {
    int dm, F, nb, C, D, d, T, nh;
};

__device__ __forceinline__ float silu_f(float z) { return z / (1.f + expf(-z)); }
__device__ __forceinline__ float silu_grad_f(float z) {
    const float s = 1.f / (1.f + expf(-z));
    return s * (1.f + z * (1.f - s));
}

// ---------------------------------------------------------------------------
// time embedding: s(tau), z1 = T1 s + tb1, phi = T2 SiLU(z1) + tb2 (one CTA
// per sample; one warp per output row, lanes along the dot product)
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_flow_time(const float* __restrict__ tau,
                                                   const int* __restrict__ sample_slot,
                                                   const __grid_constant__ FlowSlots fs, FlowDims dd,
                                                   const uint16_t* __restrict__ t1,
                                                   const uint16_t* __restrict__ tb1,
                                                   const uint16_t* __restrict__ t2,
                                                   const uint16_t* __restrict__ tb2,
                                                   float* __restrict__ sfeat,
                                                   float* __restrict__ z1, float* __restrict__ phi) {
    extern __shared__ float sh[];  // s(tau) [dm], SiLU(z1) [dm]
    const int s = blockIdx.x, dm = dd.dm, half = dm / 2;
    const int t = fs.tenant[sample_slot[s]];
    const float tv = tau[s];
    for (int i = threadIdx.x; i < dm; i += blockDim.x) {
        const int k = i < half ? i : i - half;
        const float w = powf(10000.f, -(float)k / (float)half);
        const float a = 1000.f * tv * w;
        const float v = i < half ? sinf(a) : cosf(a);
        sh[i] = v;
        sfeat[(size_t)s * dm + i] = v;
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
    const uint16_t* T1 = t1 + (size_t)t * dm * dm;
    for (int j = warp; j < dm; j += nw) {
        float acc = 0.f;
        for (int k = lane; k < dm; k += 32) acc += bf2f(T1[(size_t)j * dm + k]) * sh[k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) {
            const float z = acc + bf2f(tb1[(size_t)t * dm + j]);
            z1[(size_t)s * dm + j] = z;
            sh[dm + j] = silu_f(z);
        }
    }
    __syncthreads();
    const uint16_t* T2 = t2 + (size_t)t * dm * dm;
    for (int j = warp; j < dm; j += nw) {
        float acc = 0.f;
        for (int k = lane; k < dm; k += 32) acc += bf2f(T2[(size_t)j * dm + k]) * sh[dm + k];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) phi[(size_t)s * dm + j] = acc + bf2f(tb2[(size_t)t * dm + j]);
    }
}

// ---------------------------------------------------------------------------
// token embedding: x = tau a + (1 - tau) eps (or x given), u = a - eps,
// h = x W_in^T + b_in + pos_c + phi_s.  One CTA per action row.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_flow_embed(
    const float* __restrict__ actions, const float* __restrict__ noise,
    const float* __restrict__ tau, const float* __restrict__ xin,
    const int* __restrict__ sample_slot, const __grid_constant__ FlowSlots fs, FlowDims dd,
    const uint16_t* __restrict__ w_in, const uint16_t* __restrict__ b_in,
    const uint16_t* __restrict__ pos, const float* __restrict__ phi, float* __restrict__ x_out,
    float* __restrict__ u_out, float* __restrict__ h) {
    __shared__ float xs[kMaxD];
    const int r = blockIdx.x, C = dd.C, D = dd.D, dm = dd.dm;
    const int s = r / C, c = r % C;
    const int t = fs.tenant[sample_slot[s]];
    if (threadIdx.x < D) {
        const size_t e = (size_t)r * D + threadIdx.x;
        float x;
        if (xin) {
            x = xin[e];
        } else {
            const float tv = tau[s], a = actions[e], n = noise[e];
            x = tv * a + (1.f - tv) * n;
            u_out[e] = a - n;
        }
        xs[threadIdx.x] = x;
        x_out[e] = x;
    }
    __syncthreads();
    const uint16_t* W = w_in + (size_t)t * dm * D;
    for (int j = threadIdx.x; j < dm; j += blockDim.x) {
        float acc = bf2f(b_in[(size_t)t * dm + j]) + bf2f(pos[((size_t)t * C + c) * dm + j]) +
                    phi[(size_t)s * dm + j];
        for (int k = 0; k < D; ++k) acc += xs[k] * bf2f(W[(size_t)j * D + k]);
        h[(size_t)r * dm + j] = acc;
    }
}

// ---------------------------------------------------------------------------
// attention: per (sample, head) the C action queries against the sample's L
// context keys then its C action keys, online softmax in fp32 (log2 units).
// One thread per query; keys staged 32 at a time in shared memory.
//   qkv [M_a, 3 dm] bf16 (q | k_a | v_a), kvc [N, 2 dm] bf16 (k_c | v_c),
//   o [M_a, dm] bf16, lse [M_a, nh] fp32 (log2 of the softmax denominator
//   of the log2e-scaled scores).
// ---------------------------------------------------------------------------
constexpr int kKT = 32;  // keys per staged tile

__device__ __forceinline__ void stage_keys(float (*sk)[kHd + 1], float (*sv)[kHd + 1], int j0,
                                           int nk, int L, const uint16_t* __restrict__ kvc,
                                           int ctx0, const uint16_t* __restrict__ qkv, int act0,
                                           int dm, int h) {
    for (int i = threadIdx.x; i < kKT * kHd; i += blockDim.x) {
        const int jj = i / kHd, e = i % kHd, j = j0 + jj;
        float kv = 0.f, vv = 0.f;
        if (jj < nk) {
            if (j < L) {
                const uint16_t* row = kvc + (size_t)(ctx0 + j) * 2 * dm;
                kv = bf2f(row[h * kHd + e]);
                vv = bf2f(row[dm + h * kHd + e]);
            } else {
                const uint16_t* row = qkv + (size_t)(act0 + j - L) * 3 * dm;
                kv = bf2f(row[dm + h * kHd + e]);
                vv = bf2f(row[2 * dm + h * kHd + e]);
            }
        }
        sk[jj][e] = kv;
        sv[jj][e] = vv;
    }
}

// One CTA per (sample, head); each query's keys are split among KS = 64 / C
// threads (thread t: query t % C, keys j = t / C (mod KS) of every staged
// tile), whose partial (max, sum, accumulator) are merged at the end.
__global__ void __launch_bounds__(64) k_flow_attn_fwd(const uint16_t* __restrict__ qkv,
                                                      const uint16_t* __restrict__ kvc,
                                                      const int* __restrict__ cu, FlowDims dd,
                                                      uint16_t* __restrict__ o,
                                                      float* __restrict__ lse) {
    __shared__ float sk[kKT][kHd + 1], sv[kKT][kHd + 1];
    __shared__ float part[64][kHd + 2];  // per thread: accumulator, max, sum
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int KS = min(8, 64 / C);  // key splits per query
    const int c = threadIdx.x % C, ks = threadIdx.x / C;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C;
    const float sc = kLog2e / sqrtf((float)kHd);
    float q[kHd], acc[kHd];
    float m = -INFINITY, l = 0.f;
    const bool act = ks < KS;
    if (act) {
        const uint16_t* qr = qkv + (size_t)(act0 + c) * 3 * dm + h * kHd;
#pragma unroll
        for (int e = 0; e < kHd; ++e) {
            q[e] = bf2f(qr[e]) * sc;
            acc[e] = 0.f;
        }
    }
    const int nkeys = L + C;
    for (int j0 = 0; j0 < nkeys; j0 += kKT) {
        const int nk = min(kKT, nkeys - j0);
        __syncthreads();
        stage_keys(sk, sv, j0, nk, L, kvc, ctx0, qkv, act0, dm, h);
        __syncthreads();
        if (!act) continue;
        for (int jj = ks; jj < nk; jj += KS) {
            float a = 0.f;
#pragma unroll
            for (int e = 0; e < kHd; ++e) a += q[e] * sk[jj][e];
            if (a > m) {
                const float alpha = exp2f(m - a);
                l *= alpha;
#pragma unroll
                for (int e = 0; e < kHd; ++e) acc[e] *= alpha;
                m = a;
            }
            const float p = exp2f(a - m);
            l += p;
#pragma unroll
            for (int e = 0; e < kHd; ++e) acc[e] += p * sv[jj][e];
        }
    }
    if (act) {
#pragma unroll
        for (int e = 0; e < kHd; ++e) part[threadIdx.x][e] = acc[e];
        part[threadIdx.x][kHd] = m;
        part[threadIdx.x][kHd + 1] = l;
    }
    __syncthreads();
    if (act && ks == 0) {
        float M = -INFINITY;
        for (int k = 0; k < KS; ++k) M = fmaxf(M, part[k * C + c][kHd]);
        float Ls = 0.f;
        float w[8];
        for (int k = 0; k < KS && k < 8; ++k) {
            const float mk = part[k * C + c][kHd];
            w[k] = mk == -INFINITY ? 0.f : exp2f(mk - M);
            Ls += part[k * C + c][kHd + 1] * w[k];
        }
        const float inv = 1.f / Ls;
        uint16_t* orow = o + (size_t)(act0 + c) * dm + h * kHd;
        for (int e = 0; e < kHd; e += 2) {
            float v0 = 0.f, v1 = 0.f;
            for (int k = 0; k < KS && k < 8; ++k) {
                v0 += part[k * C + c][e] * w[k];
                v1 += part[k * C + c][e + 1] * w[k];
            }
            *reinterpret_cast<uint32_t*>(orow + e) = pack_bf2(v0 * inv, v1 * inv);
        }
        lse[(size_t)(act0 + c) * dd.nh + h] = M + log2f(Ls);
    }
}

// Backward, query side: dq_c = scale sum_j dS_cj k_j with dS = P (dP - D_c),
// dP_cj = dO_c . v_j, D_c = dO_c . o_c.  Keys split among 64 / C threads per
// query as in the forward; the partial dq are summed at the end.
__global__ void __launch_bounds__(64) k_flow_attn_bwd_q(
    const uint16_t* __restrict__ qkv, const uint16_t* __restrict__ kvc, const int* __restrict__ cu,
    FlowDims dd, const uint16_t* __restrict__ o, const float* __restrict__ dO,
    const float* __restrict__ lse, uint16_t* __restrict__ dqkv) {
    __shared__ float sk[kKT][kHd + 1], sv[kKT][kHd + 1];
    __shared__ float sq[64][kHd + 1];  // each thread's own (scaled) query row, then its dq
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int KS = min(8, 64 / C);  // key splits per query
    const int c = threadIdx.x % C, ks = threadIdx.x / C;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C;
    const float sc = 1.f / sqrtf((float)kHd);
    float g[kHd], dq[kHd];
    float Dc = 0.f, lc = 0.f;
    const bool act = ks < KS;
    float* q = sq[threadIdx.x];
    if (act) {
        const size_t r = (size_t)(act0 + c);
        const uint16_t* qr = qkv + r * 3 * dm + h * kHd;
        const uint16_t* orow = o + r * dm + h * kHd;
        const float* gr = dO + r * dm + h * kHd;
#pragma unroll
        for (int e = 0; e < kHd; ++e) {
            q[e] = bf2f(qr[e]) * sc * kLog2e;
            g[e] = gr[e];
            Dc += g[e] * bf2f(orow[e]);
            dq[e] = 0.f;
        }
        lc = lse[r * dd.nh + h];
    }
    const int nkeys = L + C;
    for (int j0 = 0; j0 < nkeys; j0 += kKT) {
        const int nk = min(kKT, nkeys - j0);
        __syncthreads();
        stage_keys(sk, sv, j0, nk, L, kvc, ctx0, qkv, act0, dm, h);
        __syncthreads();
        if (!act) continue;
        for (int jj = ks; jj < nk; jj += KS) {
            float a = 0.f, dp = 0.f;
#pragma unroll
            for (int e = 0; e < kHd; ++e) {
                a += q[e] * sk[jj][e];
                dp += g[e] * sv[jj][e];
            }
            const float ds = exp2f(a - lc) * (dp - Dc);
#pragma unroll
            for (int e = 0; e < kHd; ++e) dq[e] += ds * sk[jj][e];
        }
    }
    __syncthreads();  // every thread is done with its query row: reuse it for dq
    if (act) {
#pragma unroll
        for (int e = 0; e < kHd; ++e) q[e] = dq[e];
    }
    __syncthreads();
    if (act && ks == 0) {
        uint16_t* dr = dqkv + (size_t)(act0 + c) * 3 * dm + h * kHd;
        for (int e = 0; e < kHd; e += 2) {
            float v0 = 0.f, v1 = 0.f;
            for (int k = 0; k < KS; ++k) {
                v0 += sq[k * C + c][e];
                v1 += sq[k * C + c][e + 1];
            }
            *reinterpret_cast<uint32_t*>(dr + e) = pack_bf2(v0 * sc, v1 * sc);
        }
    }
}

// Backward, key side, one pass per gradient (DK: dk_j = scale sum_c dS_cj
// q_c; otherwise dv_j = sum_c P_cj dO_c), so each thread keeps 64
// accumulators.  One thread per key (context keys, then action keys); the
// sample's query side for the head (q, dO, lse, D) in shared memory; each
// thread's k_j (and v_j) in a padded shared row.
template <bool DK>
__global__ void __launch_bounds__(128) k_flow_attn_bwd_kv(
    const uint16_t* __restrict__ qkv, const uint16_t* __restrict__ kvc, const int* __restrict__ cu,
    FlowDims dd, const uint16_t* __restrict__ o, const float* __restrict__ dO,
    const float* __restrict__ lse, uint16_t* __restrict__ dqkv, uint16_t* __restrict__ dkvc) {
    extern __shared__ float fsm[];
    float* sq = fsm;                      // [C][kHd + 1]
    float* sg = sq + kMaxC * (kHd + 1);   // [C][kHd + 1]
    float* sl = sg + kMaxC * (kHd + 1);   // [C]
    float* sD = sl + kMaxC;               // [C]
    float* skv = sD + kMaxC;              // [128][2 kHd + 1]
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C;
    const float sc = 1.f / sqrtf((float)kHd);
    for (int i = threadIdx.x; i < C * kHd; i += blockDim.x) {
        const int c = i / kHd, e = i % kHd;
        const size_t r = (size_t)(act0 + c);
        sq[c * (kHd + 1) + e] = bf2f(qkv[r * 3 * dm + h * kHd + e]) * sc * kLog2e;
        sg[c * (kHd + 1) + e] = dO[r * dm + h * kHd + e];
    }
    __syncthreads();
    if (threadIdx.x < C) {
        const int c = threadIdx.x;
        const size_t r = (size_t)(act0 + c);
        float Dc = 0.f;
        for (int e = 0; e < kHd; ++e) Dc += sg[c * (kHd + 1) + e] * bf2f(o[r * dm + h * kHd + e]);
        sD[c] = Dc;
        sl[c] = lse[r * dd.nh + h];
    }
    __syncthreads();
    const int nkeys = L + C;
    float* mykv = skv + threadIdx.x * (2 * kHd + 1);
    for (int j = blockIdx.z * blockDim.x + threadIdx.x; j < nkeys; j += gridDim.z * blockDim.x) {
        const uint16_t* kr;
        if (j < L)
            kr = kvc + (size_t)(ctx0 + j) * 2 * dm + h * kHd;
        else
            kr = qkv + (size_t)(act0 + j - L) * 3 * dm + dm + h * kHd;
        const uint16_t* vr = kr + dm;
        for (int e = 0; e < kHd; ++e) {
            mykv[e] = bf2f(kr[e]);
            if (DK) mykv[kHd + e] = bf2f(vr[e]);
        }
        float acc[kHd];
#pragma unroll
        for (int e = 0; e < kHd; ++e) acc[e] = 0.f;
        for (int c = 0; c < C; ++c) {
            const float* qc = sq + c * (kHd + 1);
            const float* gc = sg + c * (kHd + 1);
            float a = 0.f;
#pragma unroll
            for (int e = 0; e < kHd; ++e) a += qc[e] * mykv[e];
            const float p = exp2f(a - sl[c]);
            if (DK) {
                float dp = 0.f;
#pragma unroll
                for (int e = 0; e < kHd; ++e) dp += gc[e] * mykv[kHd + e];
                const float ds = p * (dp - sD[c]);
#pragma unroll
                for (int e = 0; e < kHd; ++e) acc[e] += ds * qc[e];
            } else {
#pragma unroll
                for (int e = 0; e < kHd; ++e) acc[e] += p * gc[e];
            }
        }
        // (DK) the queries were scaled by sc log2e; dk needs sc alone
        const float f = DK ? 1.f / kLog2e : 1.f;
        uint16_t* dr;
        if (j < L)
            dr = dkvc + (size_t)(ctx0 + j) * 2 * dm + h * kHd + (DK ? 0 : dm);
        else
            dr = dqkv + (size_t)(act0 + j - L) * 3 * dm + dm + h * kHd + (DK ? 0 : dm);
#pragma unroll
        for (int e = 0; e < kHd; e += 2)
            *reinterpret_cast<uint32_t*>(dr + e) = pack_bf2(acc[e] * f, acc[e + 1] * f);
    }
}

// ---------------------------------------------------------------------------
// output: v = nf W_out^T + b_out, and (training) dv = 2 (v - u) / n_t and
// the row's sum of (v - u)^2.  One warp per action row.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_flow_out(const uint16_t* __restrict__ nf,
                                                  const int* __restrict__ sample_slot,
                                                  const __grid_constant__ FlowSlots fs, FlowDims dd,
                                                  const uint16_t* __restrict__ w_out,
                                                  const uint16_t* __restrict__ b_out,
                                                  const float* __restrict__ u, int M,
                                                  float* __restrict__ v, float* __restrict__ dv,
                                                  float* __restrict__ rowsq) {
    const int r = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (r >= M) return;
    const int dm = dd.dm, D = dd.D, C = dd.C;
    const int slot = sample_slot[r / C];
    const int t = fs.tenant[slot];
    const float nt = (float)(fs.s1[slot] - fs.s0[slot]) * C * D;
    const uint16_t* x = nf + (size_t)r * dm;
    float sq = 0.f;
    for (int k = 0; k < D; ++k) {
        const uint16_t* wr = w_out + ((size_t)t * D + k) * dm;
        float acc = 0.f;
        for (int j = lane; j < dm; j += 32) acc += bf2f(x[j]) * bf2f(wr[j]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        acc += bf2f(b_out[(size_t)t * D + k]);
        if (lane == 0) {
            const size_t e = (size_t)r * D + k;
            v[e] = acc;
            if (u) {
                const float diff = acc - u[e];
                dv[e] = 2.f * diff / nt;
                sq += diff * diff;
            }
        }
    }
    if (u && lane == 0) rowsq[r] = sq;
}

// loss[tenant] = sum of the tenant's row sums in row order / n_t.
__global__ void k_flow_loss(const __grid_constant__ FlowSlots fs, FlowDims dd,
                            const float* __restrict__ rowsq, float* __restrict__ loss) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= fs.n) return;
    float acc = 0.f;
    for (int r = fs.s0[i] * dd.C; r < fs.s1[i] * dd.C; ++r) acc += rowsq[r];
    loss[fs.tenant[i]] = acc / ((float)(fs.s1[i] - fs.s0[i]) * dd.C * dd.D);
}

// Euler step of the sampler: x += dt v.
__global__ void k_flow_euler(float* __restrict__ x, const float* __restrict__ v, float dt, int n) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) x[i] += dt * v[i];
}

// ---------------------------------------------------------------------------
// backward of the output layer
// ---------------------------------------------------------------------------
// dnf[r] = dv[r] W_out (per action row).
__global__ void __launch_bounds__(256) k_flow_out_bwd(const float* __restrict__ dv,
                                                      const int* __restrict__ sample_slot,
                                                      const __grid_constant__ FlowSlots fs,
                                                      FlowDims dd,
                                                      const uint16_t* __restrict__ w_out,
                                                      float* __restrict__ dnf) {
    const int r = blockIdx.x, dm = dd.dm, D = dd.D;
    const int t = fs.tenant[sample_slot[r / dd.C]];
    __shared__ float g[kMaxD];
    if (threadIdx.x < D) g[threadIdx.x] = dv[(size_t)r * D + threadIdx.x];
    __syncthreads();
    for (int j = threadIdx.x; j < dm; j += blockDim.x) {
        float acc = 0.f;
        for (int k = 0; k < D; ++k) acc += g[k] * bf2f(w_out[((size_t)t * D + k) * dm + j]);
        dnf[(size_t)r * dm + j] = acc;
    }
}

// dW_out[t][k, j] = sum over the tenant's rows of dv[r, k] nf[r, j];
// db_out[t][k] = sum dv[r, k].  One CTA per (slot, k); threads along j.
__global__ void __launch_bounds__(256) k_flow_out_wgrad(const float* __restrict__ dv,
                                                        const uint16_t* __restrict__ nf,
                                                        const __grid_constant__ FlowSlots fs,
                                                        FlowDims dd, float* __restrict__ gw,
                                                        float* __restrict__ gb, int add) {
    const int i = blockIdx.x, k = blockIdx.y, dm = dd.dm, D = dd.D, C = dd.C;
    const int t = fs.tenant[i];
    const int r0 = fs.s0[i] * C, r1 = fs.s1[i] * C;
    for (int j = threadIdx.x; j < dm; j += blockDim.x) {
        float acc = 0.f;
        for (int r = r0; r < r1; ++r) acc += dv[(size_t)r * D + k] * bf2f(nf[(size_t)r * dm + j]);
        float* p = gw + ((size_t)t * D + k) * dm + j;
        *p = add ? *p + acc : acc;
    }
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int r = r0; r < r1; ++r) acc += dv[(size_t)r * D + k];
        float* p = gb + (size_t)t * D + k;
        *p = add ? *p + acc : acc;
    }
}

// ---------------------------------------------------------------------------
// backward of the embedding and of the time MLP
// ---------------------------------------------------------------------------
// Per slot, thread per width column j: dW_in[t][j, :] = sum_r dh[r, j] x[r, :],
// db_in[t][j] = sum_r dh[r, j], dpos[t][c, j] = sum over samples dh[s C + c, j].
__global__ void __launch_bounds__(256) k_flow_embed_wgrad(const float* __restrict__ dh,
                                                          const float* __restrict__ x,
                                                          const __grid_constant__ FlowSlots fs,
                                                          FlowDims dd, float* __restrict__ gw,
                                                          float* __restrict__ gb,
                                                          float* __restrict__ gpos, int add) {
    const int i = blockIdx.x, dm = dd.dm, D = dd.D, C = dd.C;
    const int j = blockIdx.y * blockDim.x + threadIdx.x;
    if (j >= dm) return;
    const int t = fs.tenant[i];
    float w[kMaxD];
#pragma unroll
    for (int k = 0; k < kMaxD; ++k) w[k] = 0.f;
    float b = 0.f;
    for (int s = fs.s0[i]; s < fs.s1[i]; ++s)
        for (int c = 0; c < C; ++c) {
            const size_t r = (size_t)s * C + c;
            const float g = dh[r * dm + j];
            b += g;
#pragma unroll
            for (int k = 0; k < kMaxD; ++k)
                if (k < D) w[k] += g * x[r * D + k];
        }
#pragma unroll
    for (int k = 0; k < kMaxD; ++k)
        if (k < D) {
            float* p = gw + ((size_t)t * dm + j) * D + k;
            *p = add ? *p + w[k] : w[k];
        }
    float* pb = gb + (size_t)t * dm + j;
    *pb = add ? *pb + b : b;
    for (int c = 0; c < C; ++c) {
        float acc = 0.f;
        for (int s = fs.s0[i]; s < fs.s1[i]; ++s) acc += dh[((size_t)s * C + c) * dm + j];
        float* p = gpos + ((size_t)t * C + c) * dm + j;
        *p = add ? *p + acc : acc;
    }
}

// dphi[s, j] = sum_c dh[s C + c, j]; then dz1[s, k] = (sum_j dphi[s, j]
// T2[j, k]) SiLU'(z1[s, k]).  One CTA per sample.
__global__ void __launch_bounds__(256) k_flow_time_bwd(const float* __restrict__ dh,
                                                       const int* __restrict__ sample_slot,
                                                       const __grid_constant__ FlowSlots fs,
                                                       FlowDims dd, const uint16_t* __restrict__ t2,
                                                       const float* __restrict__ z1,
                                                       float* __restrict__ dphi,
                                                       float* __restrict__ dz1) {
    extern __shared__ float sh[];  // dphi [dm]
    const int s = blockIdx.x, dm = dd.dm, C = dd.C;
    const int t = fs.tenant[sample_slot[s]];
    for (int j = threadIdx.x; j < dm; j += blockDim.x) {
        float acc = 0.f;
        for (int c = 0; c < C; ++c) acc += dh[((size_t)s * C + c) * dm + j];
        sh[j] = acc;
        dphi[(size_t)s * dm + j] = acc;
    }
    __syncthreads();
    const uint16_t* T2 = t2 + (size_t)t * dm * dm;
    for (int k = threadIdx.x; k < dm; k += blockDim.x) {
        float acc = 0.f;
        for (int j = 0; j < dm; ++j) acc += sh[j] * bf2f(T2[(size_t)j * dm + k]);
        dz1[(size_t)s * dm + k] = acc * silu_grad_f(z1[(size_t)s * dm + k]);
    }
}

// Per slot, row j of an outer-product sum over the tenant's samples:
//   G[t][j, k] = sum_s A[s, j] f(B[s, k]),  gb[t][j] = sum_s A[s, j]
// with f = SiLU (T2: A = dphi, B = z1) or the identity (T1: A = dz1, B = s(tau)).
template <bool SILU>
__global__ void __launch_bounds__(256) k_flow_outer(const float* __restrict__ A,
                                                    const float* __restrict__ Bm,
                                                    const __grid_constant__ FlowSlots fs,
                                                    FlowDims dd, float* __restrict__ gw,
                                                    float* __restrict__ gb, int add) {
    const int i = blockIdx.x, j = blockIdx.y, dm = dd.dm;
    const int t = fs.tenant[i];
    for (int k = threadIdx.x; k < dm; k += blockDim.x) {
        float acc = 0.f;
        for (int s = fs.s0[i]; s < fs.s1[i]; ++s) {
            const float b = Bm[(size_t)s * dm + k];
            acc += A[(size_t)s * dm + j] * (SILU ? silu_f(b) : b);
        }
        float* p = gw + ((size_t)t * dm + j) * dm + k;
        *p = add ? *p + acc : acc;
    }
    if (threadIdx.x == 0) {
        float acc = 0.f;
        for (int s = fs.s0[i]; s < fs.s1[i]; ++s) acc += A[(size_t)s * dm + j];
        float* p = gb + (size_t)t * dm + j;
        *p = add ? *p + acc : acc;
    }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
constexpr size_t kAlign = 256;
size_t up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

struct FlowWs {
    int* status;
    uint16_t* ones;      // [dm] bf16 1.0 (the non-affine norm's gain)
    float *sfeat, *z1, *phi;  // [S, dm]
    float *x, *u, *v, *dv;    // [M_a, D]
    float* rowsq;             // [M_a]
    float* h;                 // [M_a, dm] the residual stream
    float* h_out;             // [M_a, dm]
    uint16_t* nf;             // [M_a, dm]
    // per block
    float *h_in, *h_mid;      // [nb][M_a, dm]
    uint16_t *n1, *n2, *o;    // [nb][M_a, dm]
    uint16_t* qkv;            // [nb][M_a, 3 dm]
    float* lse;               // [nb][M_a, nh]
    uint16_t* m;              // [nb][M_a, F]
    uint16_t* kvc;            // [nb][N, 2 dm]
    // backward scratch
    float *dh, *dn, *dO;      // [M_a, dm]
    uint16_t* dh_bf;          // [M_a, dm]
    uint16_t* gu;             // [M_a, 2 F]
    uint16_t* dqkv;           // [M_a, 3 dm]
    uint16_t* dkvc;           // [N, 2 dm]
    uint16_t* wt;             // transposed weights of one block [T, max]
    float *dphi, *dz1;        // [S, dm]
    size_t bytes;
};

FlowWs carve_flow(const FlowDims& d, int S, int N, void* base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    FlowWs w{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* r = p ? p + off : nullptr;
        off += up(bytes);
        return r;
    };
    const size_t s = std::max(S, 1), n = std::max(N, 1), Ma = s * d.C, dm = d.dm, nb = d.nb;
    auto f32 = [&](size_t c) { return reinterpret_cast<float*>(take(c * 4)); };
    auto b16 = [&](size_t c) { return reinterpret_cast<uint16_t*>(take(c * 2)); };
    w.status = reinterpret_cast<int*>(take(256));
    w.ones = b16(dm);
    w.sfeat = f32(s * dm);
    w.z1 = f32(s * dm);
    w.phi = f32(s * dm);
    w.x = f32(Ma * d.D);
    w.u = f32(Ma * d.D);
    w.v = f32(Ma * d.D);
    w.dv = f32(Ma * d.D);
    w.rowsq = f32(Ma);
    w.h = f32(Ma * dm);
    w.h_out = f32(Ma * dm);
    w.nf = b16(Ma * dm);
    w.h_in = f32(nb * Ma * dm);
    w.h_mid = f32(nb * Ma * dm);
    w.n1 = b16(nb * Ma * dm);
    w.n2 = b16(nb * Ma * dm);
    w.o = b16(nb * Ma * dm);
    w.qkv = b16(nb * Ma * 3 * dm);
    w.lse = f32(nb * Ma * d.nh);
    w.m = b16(nb * Ma * d.F);
    w.kvc = b16(nb * n * 2 * dm);
    w.dh = f32(Ma * dm);
    w.dn = f32(Ma * dm);
    w.dO = f32(Ma * dm);
    w.dh_bf = b16(Ma * dm);
    w.gu = b16(Ma * 2 * d.F);
    w.dqkv = b16(Ma * 3 * dm);
    w.dkvc = b16(n * 2 * dm);
    w.wt = b16((size_t)d.T * std::max(3 * dm * dm, 2 * (size_t)d.F * dm));
    w.dphi = f32(s * dm);
    w.dz1 = f32(s * dm);
    w.bytes = off;
    return w;
}

jnx_status check_flow(const jnx_flow_head* fh, const jnx_group* g, FlowDims& d) {
    jnx_status st;
    if ((st = check_group(g))) return st;
    if (!fh || !fh->blocks || !fh->w_in || !fh->b_in || !fh->pos || !fh->t1 || !fh->tb1 ||
        !fh->t2 || !fh->tb2 || !fh->w_out || !fh->b_out)
        return fail(JNX_ERR_INVALID_ARG, "flow: null parameter");
    d.dm = fh->d_model;
    d.F = fh->d_ff;
    d.nb = fh->n_blocks;
    d.C = fh->chunk;
    d.D = fh->action_dim;
    d.d = fh->d_in;
    d.T = fh->n_tenants;
    d.nh = d.dm / kHd;
    if (d.dm != 256 && d.dm != 512 && d.dm != 1024)
        return fail(JNX_ERR_UNSUPPORTED, "flow: d_model %d not in {256, 512, 1024}", d.dm);
    if (d.F <= 0 || d.F % 128 || d.nb < 0 || d.C < 1 || d.C > kMaxC || d.D < 1 || d.D > kMaxD ||
        d.d <= 0 || d.d % 128 || d.T <= 0)
        return fail(JNX_ERR_UNSUPPORTED, "flow: unsupported dimensions");
    if (g->n_slots > kSegMaxSlots)
        return fail(JNX_ERR_UNSUPPORTED, "flow: at most %d tenants per group", kSegMaxSlots);
    for (int i = 0; i < g->n_slots; ++i)
        if (g->h_slot_tenant[i] < 0 || g->h_slot_tenant[i] >= d.T)
            return fail(JNX_ERR_INVALID_ARG, "flow: tenant %d has no expert", g->h_slot_tenant[i]);
    for (int b = 0; b < d.nb; ++b) {
        const jnx_flow_block& B = fh->blocks[b];
        if (!B.w_qkv || !B.w_kvc || !B.w_o || !B.w_gu || !B.w_d)
            return fail(JNX_ERR_INVALID_ARG, "flow: block %d has a null weight", b);
    }
    if ((long long)g->n_samples * d.C > 0x7FFFFFFF)
        return fail(JNX_ERR_UNSUPPORTED, "flow: too many action rows");
    return JNX_OK;
}

void fill_slots(const jnx_group* g, FlowSlots& fs) {
    fs = FlowSlots{};
    fs.n = g->n_slots;
    for (int i = 0; i < g->n_slots; ++i) {
        fs.tenant[i] = g->h_slot_tenant[i];
        fs.s0[i] = g->h_seg_offsets[i];
        fs.s1[i] = g->h_seg_offsets[i + 1];
    }
}

// Segments of the action rows and of the token rows, per group slot.
struct Segs {
    std::vector<int> a0, a1, t0, t1, ten;
};

Segs make_segs(const jnx_group* g, int C) {
    Segs sg;
    for (int i = 0; i < g->n_slots; ++i) {
        const int s0 = g->h_seg_offsets[i], s1 = g->h_seg_offsets[i + 1];
        sg.a0.push_back(s0 * C);
        sg.a1.push_back(s1 * C);
        sg.t0.push_back(g->h_cu_seqlens[s0]);
        sg.t1.push_back(g->h_cu_seqlens[s1]);
        sg.ten.push_back(g->h_slot_tenant[i]);
    }
    return sg;
}

jnx_status last(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

__global__ void k_fill_bf16(uint16_t* p, int n, uint16_t v) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) p[i] = v;
}

__global__ void k_fill_f32(float* p, int n, float v) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) p[i] = v;
}

// The network from h (embedded) through the blocks to v (and, with u, dv
// and the loss); saves every block's activations.  With reuse_ctx, the
// context K/V of every block are already in the workspace.
jnx_status flow_network(const jnx_flow_head* fh, const FlowDims& d, const jnx_group* g,
                        const uint16_t* hidden, const FlowWs& w, const FlowSlots& fs,
                        const Segs& sg, bool reuse_ctx, bool train, float* loss, cudaStream_t s) {
    const int S = g->n_samples, N = g->n_tokens, Ma = S * d.C, dm = d.dm, nsl = g->n_slots;
    jnx_status st;
    for (int b = 0; b < d.nb; ++b) {
        const jnx_flow_block& B = fh->blocks[b];
        float* h_in = w.h_in + (size_t)b * Ma * dm;
        float* h_mid = w.h_mid + (size_t)b * Ma * dm;
        uint16_t* n1 = w.n1 + (size_t)b * Ma * dm;
        uint16_t* n2 = w.n2 + (size_t)b * Ma * dm;
        uint16_t* o = w.o + (size_t)b * Ma * dm;
        uint16_t* qkv = w.qkv + (size_t)b * Ma * 3 * dm;
        float* lse = w.lse + (size_t)b * Ma * d.nh;
        uint16_t* m = w.m + (size_t)b * Ma * d.F;
        uint16_t* kvc = w.kvc + (size_t)b * N * 2 * dm;
        if (cudaMemcpyAsync(h_in, w.h, (size_t)Ma * dm * 4, cudaMemcpyDeviceToDevice, s) !=
            cudaSuccess)
            return last("flow: copy");
        {
            TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 6.0, s);
            if ((st = rmsnorm_launch(w.h, w.ones, kEps, Ma, dm, n1, s))) return st;
        }
        GemmParams p{};
        p.M = Ma;
        p.N = 3 * dm;
        p.K = dm;
        p.epi = EPI_BF16;
        p.out = qkv;
        p.ldo = 3 * dm;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * 3 * dm * dm, s);
            if ((st = gemm_launch_seg(n1, dm, B.w_qkv, dm, d.T, p, nsl, sg.a0.data(), sg.a1.data(),
                                      sg.ten.data(), s)))
                return st;
        }
        if (!reuse_ctx) {
            p = GemmParams{};
            p.M = N;
            p.N = 2 * dm;
            p.K = d.d;
            p.epi = EPI_BF16;
            p.out = kvc;
            p.ldo = 2 * dm;
            p.status = w.status;
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * N * 2 * dm * d.d, s);
            if ((st = gemm_launch_seg(hidden, d.d, B.w_kvc, d.d, d.T, p, nsl, sg.t0.data(),
                                      sg.t1.data(), sg.ten.data(), s)))
                return st;
        }
        {
            double fl = 0.0;
            for (int i = 0; i < S; ++i)
                fl += 4.0 * d.C * (double)(g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i] + d.C) * dm;
            TraceScope ts(JNX_K_FLOW_ATTN, fl, s);
            k_flow_attn_fwd<<<dim3(S, d.nh), 64, 0, s>>>(qkv, kvc, g->cu_seqlens, d, o, lse);
            if ((st = last("flow attention"))) return st;
        }
        p = GemmParams{};
        p.M = Ma;
        p.N = dm;
        p.K = dm;
        p.epi = EPI_RESID;
        p.resid = w.h;
        p.ldr = dm;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * dm * dm, s);
            if ((st = gemm_launch_seg(o, dm, B.w_o, dm, d.T, p, nsl, sg.a0.data(), sg.a1.data(),
                                      sg.ten.data(), s)))
                return st;
        }
        if (cudaMemcpyAsync(h_mid, w.h, (size_t)Ma * dm * 4, cudaMemcpyDeviceToDevice, s) !=
            cudaSuccess)
            return last("flow: copy");
        {
            TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 6.0, s);
            if ((st = rmsnorm_launch(w.h, w.ones, kEps, Ma, dm, n2, s))) return st;
        }
        p = GemmParams{};
        p.M = Ma;
        p.N = 2 * d.F;
        p.K = dm;
        p.epi = EPI_GLU;
        p.out = m;
        p.ldo = d.F;
        p.act = JNX_GLU_SWIGLU;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * 2 * d.F * dm, s);
            if ((st = gemm_launch_seg(n2, dm, B.w_gu, dm, d.T, p, nsl, sg.a0.data(), sg.a1.data(),
                                      sg.ten.data(), s)))
                return st;
        }
        p = GemmParams{};
        p.M = Ma;
        p.N = dm;
        p.K = d.F;
        p.epi = EPI_RESID;
        p.resid = w.h;
        p.ldr = dm;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * dm * d.F, s);
            if ((st = gemm_launch_seg(m, d.F, B.w_d, d.F, d.T, p, nsl, sg.a0.data(), sg.a1.data(),
                                      sg.ten.data(), s)))
                return st;
        }
    }
    TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 8.0, s);
    if (cudaMemcpyAsync(w.h_out, w.h, (size_t)Ma * dm * 4, cudaMemcpyDeviceToDevice, s) !=
        cudaSuccess)
        return last("flow: copy");
    if ((st = rmsnorm_launch(w.h, w.ones, kEps, Ma, dm, w.nf, s))) return st;
    k_flow_out<<<(Ma + 7) / 8, 256, 0, s>>>(w.nf, g->sample_slot, fs, d, fh->w_out, fh->b_out,
                                            train ? w.u : nullptr, Ma, w.v, w.dv, w.rowsq);
    if ((st = last("flow output"))) return st;
    if (train && loss) {
        k_flow_loss<<<(nsl + 63) / 64, 64, 0, s>>>(fs, d, w.rowsq, loss);
        if ((st = last("flow loss"))) return st;
    }
    return JNX_OK;
}

}  // namespace
}  // namespace jnx

using namespace jnx;

extern "C" size_t jnx_flow_workspace_bytes(const jnx_flow_head* fh, const jnx_group* g) {
    if (!fh || !g) return 0;
    FlowDims d{fh->d_model, fh->d_ff, fh->n_blocks, fh->chunk, fh->action_dim, fh->d_in,
               fh->n_tenants, fh->d_model / kHd};
    return carve_flow(d, g->n_samples, g->n_tokens, nullptr).bytes;
}

static jnx_status flow_begin(const jnx_flow_head* fh, const jnx_group* g, const uint16_t* hidden,
                             void* workspace, size_t ws_bytes, FlowDims& d, FlowWs& w) {
    jnx_status st;
    if ((st = check_flow(fh, g, d))) return st;
    if (!workspace || (g->n_tokens > 0 && !hidden))
        return fail(JNX_ERR_INVALID_ARG, "flow: null workspace or hidden rows");
    w = carve_flow(d, g->n_samples, g->n_tokens, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "flow: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    return JNX_OK;
}

// time embedding + token embedding into w.h
static jnx_status flow_embed(const jnx_flow_head* fh, const FlowDims& d, const jnx_group* g,
                             const FlowWs& w, const FlowSlots& fs, const float* actions,
                             const float* noise, const float* tau, const float* xin,
                             cudaStream_t s) {
    const int S = g->n_samples, Ma = S * d.C;
    TraceScope ts(JNX_K_FLOW_MISC, (double)S * d.dm * d.dm * 4.0, s);
    k_fill_bf16<<<(d.dm + 255) / 256, 256, 0, s>>>(w.ones, d.dm, (uint16_t)0x3F80);
    k_flow_time<<<S, 256, 2 * d.dm * sizeof(float), s>>>(tau, g->sample_slot, fs, d, fh->t1,
                                                         fh->tb1, fh->t2, fh->tb2, w.sfeat, w.z1,
                                                         w.phi);
    k_flow_embed<<<Ma, 256, 0, s>>>(actions, noise, tau, xin, g->sample_slot, fs, d, fh->w_in,
                                    fh->b_in, fh->pos, w.phi, w.x, w.u, w.h);
    return last("flow embedding");
}

extern "C" jnx_status jnx_flow_forward(const jnx_flow_head* fh, const jnx_group* g,
                                       const uint16_t* hidden, const float* actions,
                                       const float* noise, const float* tau, float* velocity,
                                       float* loss, void* workspace, size_t ws_bytes,
                                       void* stream) {
    clear_error();
    FlowDims d;
    FlowWs w;
    jnx_status st;
    if ((st = flow_begin(fh, g, hidden, workspace, ws_bytes, d, w))) return st;
    if (g->n_samples == 0) return JNX_OK;
    if (!actions || !noise || !tau || !velocity || !loss)
        return fail(JNX_ERR_INVALID_ARG, "flow forward: null buffer");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    static thread_local FlowSlots fs;
    fill_slots(g, fs);
    const Segs sg = make_segs(g, d.C);
    if ((st = flow_embed(fh, d, g, w, fs, actions, noise, tau, nullptr, s))) return st;
    if ((st = flow_network(fh, d, g, hidden, w, fs, sg, false, true, loss, s))) return st;
    if (cudaMemcpyAsync(velocity, w.v, (size_t)g->n_samples * d.C * d.D * 4,
                        cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return last("flow: velocity copy");
    return JNX_OK;
}

extern "C" jnx_status jnx_flow_sample(const jnx_flow_head* fh, const jnx_group* g,
                                      const uint16_t* hidden, const float* noise, int32_t n_steps,
                                      float* actions, void* workspace, size_t ws_bytes,
                                      void* stream) {
    clear_error();
    FlowDims d;
    FlowWs w;
    jnx_status st;
    if ((st = flow_begin(fh, g, hidden, workspace, ws_bytes, d, w))) return st;
    if (n_steps < 1) return fail(JNX_ERR_INVALID_ARG, "flow sample: n_steps < 1");
    if (g->n_samples == 0) return JNX_OK;
    if (!noise || !actions) return fail(JNX_ERR_INVALID_ARG, "flow sample: null buffer");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    static thread_local FlowSlots fs;
    fill_slots(g, fs);
    const Segs sg = make_segs(g, d.C);
    const int n = g->n_samples * d.C * d.D;
    if (cudaMemcpyAsync(actions, noise, (size_t)n * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return last("flow: copy");
    // tau of step i for every sample, in the u buffer (no target when sampling)
    for (int i = 0; i < n_steps; ++i) {
        k_fill_f32<<<(g->n_samples + 255) / 256, 256, 0, s>>>(w.u, g->n_samples,
                                                             (float)i / (float)n_steps);
        if ((st = flow_embed(fh, d, g, w, fs, nullptr, nullptr, w.u, actions, s))) return st;
        if ((st = flow_network(fh, d, g, hidden, w, fs, sg, i > 0, false, nullptr, s))) return st;
        k_flow_euler<<<(n + 255) / 256, 256, 0, s>>>(actions, w.v, 1.f / (float)n_steps, n);
        if ((st = last("flow euler"))) return st;
    }
    return JNX_OK;
}

extern "C" jnx_status jnx_flow_backward(const jnx_flow_head* fh, const jnx_group* g,
                                        const uint16_t* hidden, const jnx_flow_grads* gr,
                                        int32_t accumulate, void* workspace, size_t ws_bytes,
                                        void* stream) {
    clear_error();
    FlowDims d;
    FlowWs w;
    jnx_status st;
    if ((st = flow_begin(fh, g, hidden, workspace, ws_bytes, d, w))) return st;
    if (!gr || !gr->blocks || !gr->w_in || !gr->b_in || !gr->pos || !gr->t1 || !gr->tb1 ||
        !gr->t2 || !gr->tb2 || !gr->w_out || !gr->b_out)
        return fail(JNX_ERR_INVALID_ARG, "flow backward: null gradient buffer");
    for (int b = 0; b < d.nb; ++b) {
        const jnx_flow_block_grads& G = gr->blocks[b];
        if (!G.w_qkv || !G.w_kvc || !G.w_o || !G.w_gu || !G.w_d)
            return fail(JNX_ERR_INVALID_ARG, "flow backward: block %d null gradient", b);
    }
    if (g->n_samples == 0) return JNX_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    static thread_local FlowSlots fs;
    fill_slots(g, fs);
    const Segs sg = make_segs(g, d.C);
    const int S = g->n_samples, Ma = S * d.C, dm = d.dm, F = d.F, T = d.T, nsl = g->n_slots;
    const int add = accumulate ? 1 : 0;
    static thread_local SegRows ra, rt;  // action-row and token-row segments
    ra = SegRows{};
    rt = SegRows{};
    ra.n = rt.n = nsl;
    for (int i = 0; i < nsl; ++i) {
        ra.tenant[i] = rt.tenant[i] = sg.ten[i];
        ra.r0[i] = sg.a0[i];
        ra.r1[i] = sg.a1[i];
        rt.r0[i] = sg.t0[i];
        rt.r1[i] = sg.t1[i];
    }
    // output layer
    {
        TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * d.D * 4.0, s);
        k_flow_out_wgrad<<<dim3(nsl, d.D), 256, 0, s>>>(w.dv, w.nf, fs, d, gr->w_out, gr->b_out,
                                                        add);
        k_flow_out_bwd<<<Ma, 256, 0, s>>>(w.dv, g->sample_slot, fs, d, fh->w_out, w.dn);
        if ((st = last("flow output backward"))) return st;
        if ((st = rms_bwd_launch(w.h_out, w.ones, kEps, w.dn, nullptr, Ma, dm, w.dh, w.dh_bf, s)))
            return st;
    }
    for (int b = d.nb - 1; b >= 0; --b) {
        const jnx_flow_block& B = fh->blocks[b];
        const jnx_flow_block_grads& G = gr->blocks[b];
        const float* h_in = w.h_in + (size_t)b * Ma * dm;
        const float* h_mid = w.h_mid + (size_t)b * Ma * dm;
        const uint16_t* n1 = w.n1 + (size_t)b * Ma * dm;
        const uint16_t* n2 = w.n2 + (size_t)b * Ma * dm;
        const uint16_t* o = w.o + (size_t)b * Ma * dm;
        const uint16_t* qkv = w.qkv + (size_t)b * Ma * 3 * dm;
        const float* lse = w.lse + (size_t)b * Ma * d.nh;
        const uint16_t* m = w.m + (size_t)b * Ma * F;
        const uint16_t* kvc = w.kvc + (size_t)b * g->n_tokens * 2 * dm;
        // ---- MLP: h += W_d (SiLU(g) * u) ----
        GemmParams p{};
        p.M = Ma;
        p.N = 2 * F;
        p.K = dm;
        p.epi = EPI_GLU_SAVE;
        p.out = w.gu;
        p.ldo = 2 * F;
        p.act = JNX_GLU_SWIGLU;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * 2 * F * dm, s);
            if ((st = gemm_launch_seg(n2, dm, B.w_gu, dm, T, p, nsl, sg.a0.data(), sg.a1.data(),
                                      sg.ten.data(), s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_WGRAD, 2.0 * Ma * dm * F, s);
            if ((st = seg_wgrad_launch(ra, w.dh_bf, dm, m, F, dm, F, G.w_d, (long long)dm * F,
                                       add, s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * F * dm, s);
            if ((st = transpose_launch(B.w_d, T, dm, F, w.wt, s))) return st;  // [T, F, dm]
            p = GemmParams{};
            p.M = Ma;
            p.N = F;
            p.K = dm;
            p.epi = EPI_GLU_BWD;
            p.out = w.gu;
            p.ldo = 2 * F;
            p.aux = w.gu;
            p.ldaux = 2 * F;
            p.status = w.status;
            if ((st = gemm_launch_seg(w.dh_bf, dm, w.wt, dm, T, p, nsl, sg.a0.data(),
                                      sg.a1.data(), sg.ten.data(), s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_WGRAD, 2.0 * Ma * 2 * F * dm, s);
            if ((st = seg_wgrad_launch(ra, w.gu, 2 * F, n2, dm, 2 * F, dm, G.w_gu,
                                       (long long)2 * F * dm, add, s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * dm * 2 * F, s);
            if ((st = transpose_launch(B.w_gu, T, 2 * F, dm, w.wt, s))) return st;  // [T, dm, 2F]
            p = GemmParams{};
            p.M = Ma;
            p.N = dm;
            p.K = 2 * F;
            p.epi = EPI_F32;
            p.out = w.dn;
            p.ldo = dm;
            p.status = w.status;
            if ((st = gemm_launch_seg(w.gu, 2 * F, w.wt, 2 * F, T, p, nsl, sg.a0.data(),
                                      sg.a1.data(), sg.ten.data(), s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 18.0, s);
            if ((st = rms_bwd_launch(h_mid, w.ones, kEps, w.dn, w.dh, Ma, dm, w.dh, w.dh_bf, s)))
                return st;
        }
        // ---- attention: h += o W_o^T ----
        {
            TraceScope ts(JNX_K_FLOW_WGRAD, 2.0 * Ma * dm * dm, s);
            if ((st = seg_wgrad_launch(ra, w.dh_bf, dm, o, dm, dm, dm, G.w_o, (long long)dm * dm,
                                       add, s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * dm * dm, s);
            if ((st = transpose_launch(B.w_o, T, dm, dm, w.wt, s))) return st;
            p = GemmParams{};
            p.M = Ma;
            p.N = dm;
            p.K = dm;
            p.epi = EPI_F32;
            p.out = w.dO;
            p.ldo = dm;
            p.status = w.status;
            if ((st = gemm_launch_seg(w.dh_bf, dm, w.wt, dm, T, p, nsl, sg.a0.data(),
                                      sg.a1.data(), sg.ten.data(), s)))
                return st;
        }
        {
            double fl = 0.0;
            for (int i = 0; i < S; ++i)
                fl += 8.0 * d.C * (double)(g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i] + d.C) * dm;
            TraceScope ts(JNX_K_FLOW_ATTN, fl, s);
            k_flow_attn_bwd_q<<<dim3(S, d.nh), 64, 0, s>>>(qkv, kvc, g->cu_seqlens, d, o, w.dO,
                                                           lse, w.dqkv);
            const size_t smem = (size_t)(2 * kMaxC * (kHd + 1) + 2 * kMaxC + 128 * (2 * kHd + 1)) *
                                sizeof(float);
            static bool attr = false;
            if (!attr) {
                if (cudaFuncSetAttribute(k_flow_attn_bwd_kv<true>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem) != cudaSuccess ||
                    cudaFuncSetAttribute(k_flow_attn_bwd_kv<false>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem) != cudaSuccess)
                    return last("flow: smem attribute");
                attr = true;
            }
            k_flow_attn_bwd_kv<true><<<dim3(S, d.nh, 4), 128, smem, s>>>(
                qkv, kvc, g->cu_seqlens, d, o, w.dO, lse, w.dqkv, w.dkvc);
            k_flow_attn_bwd_kv<false><<<dim3(S, d.nh, 4), 128, smem, s>>>(
                qkv, kvc, g->cu_seqlens, d, o, w.dO, lse, w.dqkv, w.dkvc);
            if ((st = last("flow attention backward"))) return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_WGRAD,
                          2.0 * Ma * 3 * dm * dm + 2.0 * g->n_tokens * 2 * dm * d.d, s);
            if ((st = seg_wgrad_launch(ra, w.dqkv, 3 * dm, n1, dm, 3 * dm, dm, G.w_qkv,
                                       (long long)3 * dm * dm, add, s)) ||
                (st = seg_wgrad_launch(rt, w.dkvc, 2 * dm, hidden, d.d, 2 * dm, d.d, G.w_kvc,
                                       (long long)2 * dm * d.d, add, s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_GEMM, 2.0 * Ma * dm * 3 * dm, s);
            if ((st = transpose_launch(B.w_qkv, T, 3 * dm, dm, w.wt, s))) return st;  // [T, dm, 3dm]
            p = GemmParams{};
            p.M = Ma;
            p.N = dm;
            p.K = 3 * dm;
            p.epi = EPI_F32;
            p.out = w.dn;
            p.ldo = dm;
            p.status = w.status;
            if ((st = gemm_launch_seg(w.dqkv, 3 * dm, w.wt, 3 * dm, T, p, nsl, sg.a0.data(),
                                      sg.a1.data(), sg.ten.data(), s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 18.0, s);
            if ((st = rms_bwd_launch(h_in, w.ones, kEps, w.dn, w.dh, Ma, dm, w.dh, w.dh_bf, s)))
                return st;
        }
    }
    // ---- embedding and time MLP ----
    TraceScope ts(JNX_K_FLOW_MISC, (double)Ma * dm * 8.0 + (double)S * dm * dm * 8.0, s);
    k_flow_embed_wgrad<<<dim3(nsl, (dm + 255) / 256), 256, 0, s>>>(w.dh, w.x, fs, d, gr->w_in,
                                                                    gr->b_in, gr->pos, add);
    k_flow_time_bwd<<<S, 256, dm * sizeof(float), s>>>(w.dh, g->sample_slot, fs, d, fh->t2, w.z1,
                                                       w.dphi, w.dz1);
    k_flow_outer<true><<<dim3(nsl, dm), 256, 0, s>>>(w.dphi, w.z1, fs, d, gr->t2, gr->tb2, add);
    k_flow_outer<false><<<dim3(nsl, dm), 256, 0, s>>>(w.dz1, w.sfeat, fs, d, gr->t1, gr->tb1, add);
    return last("flow embedding backward");
}
