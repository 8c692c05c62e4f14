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
//   (the weight gradients formed through the queries per sample:
//    dWk = Q^T (sum_s dS_s^T X_s) / sqrt(dq), dWv = sum_s dO_s^T (P_s^T X_s))
// Loss (both): l_t = sum (y - t)^2 / (n_t * width), dy = 2 (y - t) / (n_t width).
// All sums run in a fixed order inside one thread, one CTA or one
// tensor-core instruction sequence (no atomics), so a tenant's results are
// identical whether it runs grouped or alone.
#include <type_traits>

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

// Where a gradient kernel finishes a parameter's gradient element.  With
// NoOpt it is stored into the slot's gradient buffer (added to it when the
// slot accumulates); with HeadOptTable the element (plus the buffer's
// accumulated value) goes straight into the tenant's AdamW update, and the
// moments, fp32 master and bf16 parameter are rewritten instead.
struct NoOpt {};
template <class OT>
constexpr bool kFused = std::is_same<OT, HeadOptTable>::value;

__device__ __forceinline__ void opt_step1(const HeadOpt& o, int k, size_t i, float g,
                                          const AdamHp& hp) {
    float m = o.m[k][i], v = o.v[k][i];
    const float p = adamw_elem(g, m, v, o.master[k][i], o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps,
                               hp.wd);
    o.m[k][i] = m;
    o.v[k][i] = v;
    o.master[k][i] = p;
    o.p[k][i] = f2bf(p);
}

// four consecutive elements i .. i + 3 (i a multiple of 4; 16-byte state)
__device__ __forceinline__ void opt_step4(const HeadOpt& o, int k, size_t i, float4 g,
                                          const AdamHp& hp) {
    float4 m = *reinterpret_cast<const float4*>(o.m[k] + i);
    float4 v = *reinterpret_cast<const float4*>(o.v[k] + i);
    float4 p = *reinterpret_cast<const float4*>(o.master[k] + i);
    p.x = adamw_elem(g.x, m.x, v.x, p.x, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    p.y = adamw_elem(g.y, m.y, v.y, p.y, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    p.z = adamw_elem(g.z, m.z, v.z, p.z, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    p.w = adamw_elem(g.w, m.w, v.w, p.w, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    *reinterpret_cast<float4*>(o.m[k] + i) = m;
    *reinterpret_cast<float4*>(o.v[k] + i) = v;
    *reinterpret_cast<float4*>(o.master[k] + i) = p;
    *reinterpret_cast<uint2*>(o.p[k] + i) = make_uint2(pack_bf2(p.x, p.y), pack_bf2(p.z, p.w));
}

// two consecutive elements i, i + 1 (i even; 8-byte state)
__device__ __forceinline__ void opt_step2(const HeadOpt& o, int k, size_t i, float2 g,
                                          const AdamHp& hp) {
    float2 m = *reinterpret_cast<const float2*>(o.m[k] + i);
    float2 v = *reinterpret_cast<const float2*>(o.v[k] + i);
    float2 p = *reinterpret_cast<const float2*>(o.master[k] + i);
    p.x = adamw_elem(g.x, m.x, v.x, p.x, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    p.y = adamw_elem(g.y, m.y, v.y, p.y, o.c1, o.c2, hp.lr, hp.b1, hp.b2, hp.eps, hp.wd);
    *reinterpret_cast<float2*>(o.m[k] + i) = m;
    *reinterpret_cast<float2*>(o.v[k] + i) = v;
    *reinterpret_cast<float2*>(o.master[k] + i) = p;
    *reinterpret_cast<uint32_t*>(o.p[k] + i) = pack_bf2(p.x, p.y);
}

// ---------------------------------------------------------------------------
// Segmented linear layer: out[s, j] = sum_k in[s, k] W[j, k] + b[j] over the
// slot's samples, on the bf16 tensor cores (mma.sync m16n8k16, fp32
// accumulation).  One CTA per (8 samples, 32 output columns, slot); the
// sample block varies fastest in the grid, so the CTAs that read one weight
// tile run together and share it through L2.  K is streamed in 256-column
// chunks through a ring of kLinStages shared-memory slots (the block's 32
// weight rows and its samples' input rows, by cp.async, kLinStages - 1
// chunks ahead of the arithmetic).  W is bf16 already; the fp32 inputs enter
// as two bf16 operands, hi = bf16(x) and lo = bf16(x - hi), so W x = W hi +
// W lo to about 2^-17 of x.  Warp w takes the chunk's columns 32 w .. + 31
// (two 16-deep steps) for all 32 output columns (two 16-row tiles) and the 8
// samples; the 8 warps' partial sums are added in warp order at the end, so
// the result does not depend on the group around the slot.
//   LAYER 1: MLP first layer (W1, b1; in = pooled); stores z and h = SiLU(z).
//   LAYER 2: output layer of either head (W2 or Wout; in = h); stores y and
//            scatters it to the caller's predictions at each target offset.
// ---------------------------------------------------------------------------
constexpr int kLinCols = 32, kLinS = 8, kLinK = 256;
constexpr int kLinStages = 4;
constexpr int kLinWPad = kLinK + 8;  // weight row stride (bf16): conflict-free ldmatrix
constexpr int kLinXPad = kLinK + 8;  // input row stride (fp32): conflict-free 8-byte loads
constexpr int kLinWBytes = kLinCols * kLinWPad * 2;
constexpr int kLinXBytes = kLinS * kLinXPad * 4;
constexpr int kLinSmem = kLinStages * (kLinWBytes + kLinXBytes);
constexpr int kLinRedPad = kLinCols + 4;  // [warp][sample][column] partial sums
static_assert(8 * kLinS * kLinRedPad * 4 <= kLinSmem, "partial sums reuse the ring");

template <int LAYER>
__global__ void __launch_bounds__(256, 2) k_head_lin(const __grid_constant__ HeadTable tab,
                                                  const float* __restrict__ in, int ld_in,
                                                  float* __restrict__ z_out, float* __restrict__ h_out,
                                                  int ld_out, const int* __restrict__ sample_target,
                                                  float* __restrict__ preds) {
    extern __shared__ __align__(16) uint8_t lin_smem[];
    const HeadSlot& hs = tab.slot[blockIdx.z];
    if (LAYER == 1 && hs.kind != JNX_HEAD_MLP) return;
    const int J = LAYER == 1 ? hs.hid : hs.width;
    const int K = LAYER == 1 ? hs.d_in : hs.hid;
    const uint16_t* W = LAYER == 1 ? hs.w1 : hs.w2;
    const uint16_t* B = LAYER == 1 ? hs.b1 : hs.b2;
    const int j0 = blockIdx.y * kLinCols, s0 = hs.s0 + blockIdx.x * kLinS;
    if (j0 >= J || s0 >= hs.s1) return;
    const int ns = min(kLinS, hs.s1 - s0);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    auto sw = [&](int b) { return reinterpret_cast<uint16_t*>(lin_smem + b * kLinWBytes); };
    auto sx = [&](int b) {
        return reinterpret_cast<float*>(lin_smem + kLinStages * kLinWBytes + b * kLinXBytes);
    };
    const int nch = (K + kLinK - 1) / kLinK;
    // chunk kc into ring slot kc % kLinStages, zero-filled past J, K or the
    // slot's samples; one commit group per chunk (empty past the last one)
    auto stage = [&](int kc) {
        if (kc < nch) {
            const int b = kc % kLinStages, k0 = kc * kLinK, nk = min(kLinK, K - k0);
            uint16_t* w = sw(b);
            for (int i = threadIdx.x; i < kLinCols * (kLinK / 8); i += 256) {
                const int c = i / (kLinK / 8), u = i % (kLinK / 8);
                const bool ok = j0 + c < J && 8 * u < nk;
                cp_async16(smem_u32(w + c * kLinWPad + 8 * u),
                           ok ? (const void*)(W + (size_t)(j0 + c) * K + k0 + 8 * u)
                              : (const void*)W,
                           ok);
            }
            float* x = sx(b);
            for (int i = threadIdx.x; i < kLinS * (kLinK / 4); i += 256) {
                const int r = i / (kLinK / 4), u = i % (kLinK / 4);
                const bool ok = r < ns && 4 * u < nk;
                cp_async16(smem_u32(x + r * kLinXPad + 4 * u),
                           ok ? (const void*)(in + (size_t)(s0 + r) * ld_in + k0 + 4 * u)
                              : (const void*)in,
                           ok);
            }
        }
        cp_async_commit();
    };
    // acc[row tile m][e]: output column j0 + 16 m + lane / 4 (+ 8 for e >= 2),
    // sample 2 (lane % 4) (+ 1 for odd e)
    float acc[2][4];
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[m][e] = 0.f;
    const int g = lane >> 2, q = lane & 3;
#pragma unroll
    for (int kc = 0; kc < kLinStages - 1; ++kc) stage(kc);
    for (int kc = 0; kc < nch; ++kc) {
        // chunk kc landed (kLinStages - 1 groups were committed after it), and
        // every warp is done with chunk kc - 1, whose slot is refilled next
        cp_async_wait<kLinStages - 2>();
        __syncthreads();
        stage(kc + kLinStages - 1);
        const int b = kc % kLinStages;
        const uint16_t* ws = sw(b);
        const float* xs = sx(b);
#pragma unroll
        for (int st = 0; st < 2; ++st) {
            const int kb = 32 * warp + 16 * st;
            // B (16 deep x 8 samples): sample g, depths 2q, 2q + 1 and 2q + 8, 2q + 9
            const float2 x0 = *reinterpret_cast<const float2*>(xs + g * kLinXPad + kb + 2 * q);
            const float2 x1 = *reinterpret_cast<const float2*>(xs + g * kLinXPad + kb + 2 * q + 8);
            const uint32_t h0 = pack_bf2(x0.x, x0.y), h1 = pack_bf2(x1.x, x1.y);
            const uint32_t l0 = pack_bf2(x0.x - bf2f((uint16_t)(h0 & 0xffff)),
                                         x0.y - bf2f((uint16_t)(h0 >> 16)));
            const uint32_t l1 = pack_bf2(x1.x - bf2f((uint16_t)(h1 & 0xffff)),
                                         x1.y - bf2f((uint16_t)(h1 >> 16)));
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                uint32_t a[4];
                const int r = 16 * m + (lane & 7) + ((lane >> 3) & 1) * 8;
                ldsm_x4(smem_u32(ws + r * kLinWPad + kb + (lane >> 4) * 8), a[0], a[1], a[2], a[3]);
                mma_bf16(acc[m], a[0], a[1], a[2], a[3], h0, h1);
                mma_bf16(acc[m], a[0], a[1], a[2], a[3], l0, l1);
            }
        }
    }
    cp_async_wait<0>();
    __syncthreads();  // the ring is free: it takes the warps' partial sums
    float* red = reinterpret_cast<float*>(lin_smem);
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int e = 0; e < 4; ++e)
            red[(warp * kLinS + 2 * q + (e & 1)) * kLinRedPad + 16 * m + g + 8 * (e >> 1)] =
                acc[m][e];
    __syncthreads();
    const int i = threadIdx.x >> 5, j = j0 + lane;  // sample s0 + i, column j
    if (i < ns && j < J) {
        float sum = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) sum += red[(w * kLinS + i) * kLinRedPad + lane];
        const int s = s0 + i;
        const float zz = sum + bf2f(B[j]);
        z_out[(size_t)s * ld_out + j] = zz;
        if (LAYER == 1)
            h_out[(size_t)s * ld_out + j] = silu_f(zz);
        else
            preds[sample_target[s] + j] = zz;
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
// db[o] = sum_s dy[s, o], over the slot's samples in order.  One CTA per
// (slot, 16 outputs o, 256 columns j); a thread keeps 4 o x 4 j; the
// samples' dy and h rows are staged 32 at a time in shared memory.
template <class OT>
__global__ void __launch_bounds__(256) k_head_dw_out(const __grid_constant__ HeadTable tab,
                                                     const __grid_constant__ OT opt, AdamHp hp,
                                                     const float* __restrict__ dy, int ld_y,
                                                     const float* __restrict__ h, int ld_h) {
    __shared__ __align__(16) float sh[32][256];
    __shared__ __align__(16) float sd[32][16];
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int o0 = blockIdx.y * 16, jb = blockIdx.z * 256;
    if (o0 >= hs.width || jb >= hs.hid) return;
    const int ty = threadIdx.x >> 6, tx = threadIdx.x & 63;
    const int ob = o0 + 4 * ty, j0 = jb + 4 * tx;
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a) acc[a][0] = acc[a][1] = acc[a][2] = acc[a][3] = 0.f;
    for (int sb = hs.s0; sb < hs.s1; sb += 32) {
        const int nsb = min(32, hs.s1 - sb);
        __syncthreads();
        for (int i = threadIdx.x; i < 32 * 64; i += 256) {
            const int r = i >> 6, u = i & 63;
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (r < nsb && jb + 4 * u < hs.hid)
                v = *reinterpret_cast<const float4*>(h + (size_t)(sb + r) * ld_h + jb + 4 * u);
            *reinterpret_cast<float4*>(&sh[r][4 * u]) = v;
        }
        for (int i = threadIdx.x; i < 32 * 16; i += 256) {
            const int r = i >> 4, o = i & 15;
            sd[r][o] = (r < nsb && o0 + o < hs.width) ? dy[(size_t)(sb + r) * ld_y + o0 + o] : 0.f;
        }
        __syncthreads();
        for (int r = 0; r < nsb; ++r) {
            const float4 d4 = *reinterpret_cast<const float4*>(&sd[r][4 * ty]);
            const float4 x4 = *reinterpret_cast<const float4*>(&sh[r][4 * tx]);
            const float d[4] = {d4.x, d4.y, d4.z, d4.w}, x[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][e] = fmaf(d[a], x[e], acc[a][e]);
        }
    }
    if (j0 < hs.hid) {
#pragma unroll
        for (int a = 0; a < 4; ++a) {
            const int o = ob + a;
            if (o >= hs.width) break;
            float4* dst = reinterpret_cast<float4*>(hs.g_w2 + (size_t)o * hs.hid + j0);
            float4 v = make_float4(acc[a][0], acc[a][1], acc[a][2], acc[a][3]);
            if (hs.accum) {
                const float4 old = *dst;
                v.x += old.x;
                v.y += old.y;
                v.z += old.z;
                v.w += old.w;
            }
            if constexpr (kFused<OT>)
                opt_step4(opt.slot[blockIdx.x], hs.kind == JNX_HEAD_MLP ? 2 : 7,
                          (size_t)o * hs.hid + j0, v, hp);
            else
                *dst = v;
        }
    }
    if (blockIdx.z == 0 && threadIdx.x < 16 && o0 + (int)threadIdx.x < hs.width) {
        const int o = o0 + threadIdx.x;
        float accb = 0.f;
        for (int s = hs.s0; s < hs.s1; ++s) accb += dy[(size_t)s * ld_y + o];
        const float gb = hs.accum ? hs.g_b2[o] + accb : accb;
        if constexpr (kFused<OT>)
            opt_step1(opt.slot[blockIdx.x], hs.kind == JNX_HEAD_MLP ? 3 : 8, o, gb, hp);
        else
            hs.g_b2[o] = gb;
    }
}

// Gradient into the output layer's input: dh[s, j] = (sum_o dy[s, o] W[o, j])
// times SiLU'(z[s, j]) for an MLP slot (dz), plain for a query head (dO).
// One CTA per (slot, 1024 columns j, 8 samples); a thread keeps 4
// consecutive columns x 8 samples, so each weight row is read once per 8
// samples (8-byte loads); dy is staged 64 outputs at a time in shared
// memory; the outputs o are summed in order.
__global__ void __launch_bounds__(256) k_head_back_in(const __grid_constant__ HeadTable tab,
                                                      const float* __restrict__ dy, int ld_y,
                                                      const float* __restrict__ z, int ld_h,
                                                      float* __restrict__ dh) {
    __shared__ __align__(16) float sdy[64][8];
    const HeadSlot& hs = tab.slot[blockIdx.x];
    const int s0 = hs.s0 + blockIdx.z * 8, jb = blockIdx.y * 1024;
    if (s0 >= hs.s1 || jb >= hs.hid) return;
    const int ns = min(8, hs.s1 - s0);
    const int j0 = jb + 4 * threadIdx.x;
    const bool colok = j0 < hs.hid;
    float acc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
    for (int o0 = 0; o0 < hs.width; o0 += 64) {
        const int no = min(64, hs.width - o0);
        __syncthreads();
        for (int i = threadIdx.x; i < 64 * 8; i += 256) {
            const int si = i >> 6, o = i & 63;
            sdy[o][si] = (o < no && si < ns) ? dy[(size_t)(s0 + si) * ld_y + o0 + o] : 0.f;
        }
        __syncthreads();
        if (colok) {
            for (int o = 0; o < no; ++o) {
                const uint2 wv =
                    *reinterpret_cast<const uint2*>(hs.w2 + (size_t)(o0 + o) * hs.hid + j0);
                const float w[4] = {__uint_as_float(wv.x << 16), __uint_as_float(wv.x & 0xFFFF0000u),
                                    __uint_as_float(wv.y << 16), __uint_as_float(wv.y & 0xFFFF0000u)};
                const float4 da = *reinterpret_cast<const float4*>(&sdy[o][0]);
                const float4 db = *reinterpret_cast<const float4*>(&sdy[o][4]);
                const float d[8] = {da.x, da.y, da.z, da.w, db.x, db.y, db.z, db.w};
#pragma unroll
                for (int i = 0; i < 8; ++i)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[i][e] = fmaf(d[i], w[e], acc[i][e]);
            }
        }
    }
    if (!colok) return;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        if (i >= ns) break;
        const size_t at = (size_t)(s0 + i) * ld_h + j0;
        float4 v = make_float4(acc[i][0], acc[i][1], acc[i][2], acc[i][3]);
        if (hs.kind == JNX_HEAD_MLP) {
            const float4 zz = *reinterpret_cast<const float4*>(z + at);
            v.x *= silu_grad_f(zz.x);
            v.y *= silu_grad_f(zz.y);
            v.z *= silu_grad_f(zz.z);
            v.w *= silu_grad_f(zz.w);
        }
        *reinterpret_cast<float4*>(dh + at) = v;
    }
}

// MLP first-layer gradient: dW1[j, k] = sum_s dz[s, j] p[s, k]; db1[j] = sum_s dz[s, j].
// One CTA per (slot, kDw1Rows rows j, 1024-column block); a thread holds
// float4 columns of the block's rows, so each feature load serves all of
// them, and the loop over the slot's samples (in order, per element) is
// unrolled so that several samples' loads are in flight.
constexpr int kDw1Rows = 8;

template <class OT>
__global__ void __launch_bounds__(256) k_mlp_dw1(const __grid_constant__ HeadTable tab,
                                                 const __grid_constant__ OT opt, AdamHp hp,
                                                 const float* __restrict__ dz, int ld,
                                                 const float* __restrict__ p, int ld_p) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_MLP) return;
    const int j0 = blockIdx.y * kDw1Rows;
    if (j0 >= hs.hid) return;
    const int nj = min(kDw1Rows, hs.hid - j0);
    const int k4 = blockIdx.z * 256 + threadIdx.x;
    if (k4 * 4 < hs.d_in) {
        float4 acc[kDw1Rows];
#pragma unroll
        for (int r = 0; r < kDw1Rows; ++r) acc[r] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
        for (int s = hs.s0; s < hs.s1; ++s) {
            const float4 x = *reinterpret_cast<const float4*>(p + (size_t)s * ld_p + k4 * 4);
            const float* g = dz + (size_t)s * ld + j0;
#pragma unroll
            for (int r = 0; r < kDw1Rows; ++r) {
                const float gr = r < nj ? g[r] : 0.f;
                acc[r].x += gr * x.x;
                acc[r].y += gr * x.y;
                acc[r].z += gr * x.z;
                acc[r].w += gr * x.w;
            }
        }
#pragma unroll
        for (int r = 0; r < kDw1Rows; ++r) {
            if (r >= nj) break;
            const size_t at = (size_t)(j0 + r) * hs.d_in + k4 * 4;
            float4 a = acc[r];
            if (hs.accum) {
                const float4 old = *reinterpret_cast<const float4*>(hs.g_w1 + at);
                a.x += old.x;
                a.y += old.y;
                a.z += old.z;
                a.w += old.w;
            }
            if constexpr (kFused<OT>)
                opt_step4(opt.slot[blockIdx.x], 0, at, a, hp);
            else
                *reinterpret_cast<float4*>(hs.g_w1 + at) = a;
        }
    }
    if (blockIdx.z == 0 && threadIdx.x < nj) {
        const int j = j0 + threadIdx.x;
        float accb = 0.f;
        for (int s = hs.s0; s < hs.s1; ++s) accb += dz[(size_t)s * ld + j];
        const float gb = hs.accum ? hs.g_b1[j] + accb : accb;
        if constexpr (kFused<OT>)
            opt_step1(opt.slot[blockIdx.x], 1, j, gb, hp);
        else
            hs.g_b1[j] = gb;
    }
}

constexpr int kMaxQ = 32;
constexpr int kXRows = 32;   // key rows staged at a time
constexpr int kXCols = 256;  // columns per pass of the products over keys
constexpr int kXPad = 40;    // row stride (bf16) of the [query][key] / [key][query] tiles

// Shared memory of the per-sample query-head kernels: bf16 operand tiles of
// the bf16 tensor cores (mma.sync m16n8k16, fp32 accumulation), rows padded
// by 8 elements (16 bytes) so that the eight rows one ldmatrix reads fall in
// distinct banks.  fp32 operands enter as two bf16 planes, hi = bf16(x) and
// lo = bf16(x - hi) (x = hi + lo to about 2^-17 of x); a product of two split
// operands takes hi hi + hi lo + lo hi, of a split and a bf16 one hi + lo.
//   sQ [kMaxQ][dq + 8]        the learned queries (bf16, rows past nq zero)
//   sA [2][kMaxQ][dq + 8]     dO, hi and lo (backward)
//   sR [2][kXRows][dq + 8]    a chunk of key or value rows, hi and lo
//   sT [2][2][kMaxQ][kXPad]   a chunk of P / dS, query-major, hi and lo
//   sU [2][2][kXRows][kXPad]  the same chunk key-major (backward)
__host__ __device__ constexpr size_t xattn_smem_bytes(int dq, bool bwd) {
    return ((size_t)(bwd ? 3 : 1) * kMaxQ * (dq + 8) + (size_t)2 * kXRows * (dq + 8) +
            (size_t)(bwd ? 8 : 4) * kMaxQ * kXPad) *
           2;
}

// hi and lo planes of four fp32 values, packed in bf16 pairs.
__device__ __forceinline__ void split4(const float4 v, uint2& hi, uint2& lo) {
    hi = make_uint2(pack_bf2(v.x, v.y), pack_bf2(v.z, v.w));
    lo = make_uint2(pack_bf2(v.x - bf2f((uint16_t)(hi.x & 0xffff)),
                             v.y - bf2f((uint16_t)(hi.x >> 16))),
                    pack_bf2(v.z - bf2f((uint16_t)(hi.y & 0xffff)),
                             v.w - bf2f((uint16_t)(hi.y >> 16))));
}

// Rows [row0, row0 + nr) x columns [c0, c0 + nc) of the fp32 matrix R
// (stride ld) into the hi plane dst and the lo plane dst + rows * ldt (row
// stride ldt); rows nr .. rows - 1 are zero.  16-byte loads: R, ld and c0
// 16-byte aligned.
__device__ __forceinline__ void xattn_split_rows(uint16_t* dst, int rows, int ldt,
                                                 const float* __restrict__ R, int ld, size_t row0,
                                                 int nr, int c0, int nc) {
    const int units = nc / 4;
    for (int i = threadIdx.x; i < rows * units; i += blockDim.x) {
        const int r = i / units, u = i % units;
        float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
        if (r < nr) v = *reinterpret_cast<const float4*>(R + (row0 + r) * ld + c0 + 4 * u);
        uint2 hi, lo;
        split4(v, hi, lo);
        *reinterpret_cast<uint2*>(dst + (size_t)r * ldt + 4 * u) = hi;
        *reinterpret_cast<uint2*>(dst + (size_t)(rows + r) * ldt + 4 * u) = lo;
    }
}

// Keys [j0, j0 + nr) of the key-major [L][nq] block X (P or dS) into hi / lo
// planes of a query-major tile tq[plane][q][j] and, if tk, a key-major tile
// tk[plane][j][q]; entries past nr or nq are zero.
__device__ __forceinline__ void xattn_split_chunk(uint16_t* tq, uint16_t* tk,
                                                  const float* __restrict__ X, int j0, int nr,
                                                  int nq) {
    for (int i = threadIdx.x; i < kMaxQ * kXRows; i += blockDim.x) {
        const int q = i & 31, j = i >> 5;  // a key's nq values are contiguous
        const bool ok = j < nr && q < nq;
        const float x = ok ? X[(size_t)(j0 + j) * nq + q] : 0.f;
        const uint16_t hi = f2bf(x), lo = f2bf(x - bf2f(hi));
        if (tq) {
            tq[q * kXPad + j] = hi;
            tq[(kMaxQ + q) * kXPad + j] = lo;
        }
        if (tk) {
            tk[j * kXPad + q] = hi;
            tk[(kXRows + j) * kXPad + q] = lo;
        }
    }
}

// The learned queries (bf16 [nq][dq], 16-byte aligned) into sQ.
__device__ __forceinline__ void xattn_stage_q(uint16_t* sQ, int ldr, const uint16_t* __restrict__ q,
                                              int nq, int dq) {
    const int units = dq / 8;
    for (int i = threadIdx.x; i < kMaxQ * units; i += blockDim.x) {
        const int r = i / units, u = i % units;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r < nq) v = *reinterpret_cast<const uint4*>(q + (size_t)r * dq + 8 * u);
        *reinterpret_cast<uint4*>(sQ + (size_t)r * ldr + 8 * u) = v;
    }
}

// out[j * nq + q] = scale * sum_c A[q, c] R[r0 + j, c] over the sample's L
// key rows, key-major: A = (ahi, alo) split, or bf16 ahi alone (alo null).
// Per 32-key chunk (rows split into sR), warp w takes query tile w % 2 and
// keys 8 (w / 2) .. + 7, over all dq.  Ends with a barrier.
__device__ void xattn_scores(const uint16_t* ahi, const uint16_t* alo, int ldr, uint16_t* sR,
                             const float* __restrict__ R, int ldkv, int r0, int L, int nq, int dq,
                             float scale, float* __restrict__ out) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m = warp & 1, nt = warp >> 1, g = lane >> 2, t = lane & 3;
    const int arow = 16 * m + (lane & 7) + ((lane >> 3) & 1) * 8, acol = (lane >> 4) * 8;
    // B (8 keys x 16 deep): matrices hi / k 0-7, hi / k 8-15, lo / k 0-7, lo / k 8-15
    const int brow = 8 * nt + (lane & 7), bcol = ((lane >> 3) & 1) * 8;
    const uint16_t* bsrc = sR + (size_t)(lane >> 4) * kXRows * ldr + (size_t)brow * ldr + bcol;
    for (int j0 = 0; j0 < L; j0 += kXRows) {
        const int nr = min(kXRows, L - j0);
        __syncthreads();  // the previous chunk's readers (or the A tiles' writers) done
        xattn_split_rows(sR, kXRows, ldr, R, ldkv, (size_t)r0 + j0, nr, 0, dq);
        __syncthreads();
        float acc[4] = {0.f, 0.f, 0.f, 0.f};
        for (int kc = 0; kc < dq; kc += 16) {
            uint32_t a[4], b[4];
            ldsm_x4(smem_u32(ahi + (size_t)arow * ldr + kc + acol), a[0], a[1], a[2], a[3]);
            ldsm_x4(smem_u32(bsrc + kc), b[0], b[1], b[2], b[3]);
            mma_bf16(acc, a[0], a[1], a[2], a[3], b[0], b[1]);
            mma_bf16(acc, a[0], a[1], a[2], a[3], b[2], b[3]);
            if (alo) {
                ldsm_x4(smem_u32(alo + (size_t)arow * ldr + kc + acol), a[0], a[1], a[2], a[3]);
                mma_bf16(acc, a[0], a[1], a[2], a[3], b[0], b[1]);
            }
        }
        // element e: query 16 m + g (+ 8 for e >= 2), key 8 nt + 2 t (+ 1 for odd e)
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const int q = 16 * m + g + 8 * (e >> 1), key = 8 * nt + 2 * t + (e & 1);
            if (key < nr && q < nq) out[(size_t)(j0 + key) * nq + q] = acc[e] * scale;
        }
    }
    __syncthreads();
}

// acc[m][n] += X R over one staged 32-key chunk: X the query-major split
// tile tq (hi, lo planes), R the key-row split tile sR (row stride
// kXCols + 8); warp w takes columns 32 w .. + 31 (four 8-column tiles n)
// of both query tiles m.
__device__ __forceinline__ void xattn_chunk_xr(float (&acc)[2][4][4], const uint16_t* tq,
                                               const uint16_t* sR) {
    constexpr int ldt = kXCols + 8;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int kr = (lane & 7) + ((lane >> 3) & 1) * 8, arow = kr, acol = (lane >> 4) * 8;
#pragma unroll
    for (int k0 = 0; k0 < kXRows; k0 += 16) {
        uint32_t ah[2][4], al[2][4];
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            const uint16_t* a = tq + (size_t)(16 * m + arow) * kXPad + k0 + acol;
            ldsm_x4(smem_u32(a), ah[m][0], ah[m][1], ah[m][2], ah[m][3]);
            ldsm_x4(smem_u32(a + kMaxQ * kXPad), al[m][0], al[m][1], al[m][2], al[m][3]);
        }
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
            const uint16_t* b = sR + (size_t)(k0 + kr) * ldt + 32 * warp + 16 * hf + acol;
            uint32_t bh[4], bl[4];
            ldsm_x4_t(smem_u32(b), bh[0], bh[1], bh[2], bh[3]);
            ldsm_x4_t(smem_u32(b + kXRows * ldt), bl[0], bl[1], bl[2], bl[3]);
#pragma unroll
            for (int m = 0; m < 2; ++m)
#pragma unroll
                for (int n = 0; n < 2; ++n) {
                    float(&c)[4] = acc[m][2 * hf + n];
                    mma_bf16(c, ah[m][0], ah[m][1], ah[m][2], ah[m][3], bh[2 * n], bh[2 * n + 1]);
                    mma_bf16(c, ah[m][0], ah[m][1], ah[m][2], ah[m][3], bl[2 * n], bl[2 * n + 1]);
                    mma_bf16(c, al[m][0], al[m][1], al[m][2], al[m][3], bh[2 * n], bh[2 * n + 1]);
                }
        }
    }
}

// Per-query reductions over the sample's key-major [L, nq] block X (and Y):
// thread (q = tid % 32, part = tid / 32) covers keys part, part + 8, ...;
// the eight parts are combined in order.  red: 8 x 32 floats of shared
// memory.  MAX: max_j X; otherwise sum_j X * Y (Y may be X's weights).
template <bool MAX>
__device__ float xattn_reduce_q(const float* __restrict__ X, const float* __restrict__ Y, int L,
                                int nq, float* red) {
    const int q = threadIdx.x & 31, part = threadIdx.x >> 5;
    float v = MAX ? -INFINITY : 0.f;
    if (q < nq)
        for (int j = part; j < L; j += 8) {
            const float x = X[(size_t)j * nq + q];
            v = MAX ? fmaxf(v, x) : fmaf(x, Y[(size_t)j * nq + q], v);
        }
    red[part * 32 + q] = v;
    __syncthreads();
    float r = MAX ? -INFINITY : 0.f;
    for (int p = 0; p < 8; ++p) r = MAX ? fmaxf(r, red[p * 32 + q]) : r + red[p * 32 + q];
    __syncthreads();  // red is reused by the caller
    return r;  // valid in threads with q < nq (every part holds the same value)
}

// ---------------------------------------------------------------------------
// Query head, per sample.  One CTA per packed sample of a query-head slot.
// P (normalised attention) for sample s is stored key-major at P + nq * cu[s]:
// element (query q, key j) at j * nq + q (nq a multiple of 4).  The
// products run on the bf16 tensor cores with split fp32 operands (see
// xattn_smem_bytes); every sum runs in a fixed order, so a sample's result
// does not depend on the batch around it.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_xattn_fwd(const __grid_constant__ HeadTable tab, int g0,
                                                   const int* __restrict__ cu,
                                                   const int* __restrict__ sample_slot,
                                                   int sample0, const float* __restrict__ kbuf,
                                                   const float* __restrict__ vbuf, int ldkv,
                                                   float* __restrict__ P, float* __restrict__ h,
                                                   int ld_h) {
    static_assert(kMaxQ == 32 && kXRows == 32, "two 16-row tiles of queries and of keys");
    extern __shared__ __align__(16) uint8_t xsm[];
    __shared__ float red[8 * 32];
    const int s = sample0 + blockIdx.x;
    const HeadSlot& hs = tab.slot[sample_slot[s] - g0];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, dq = hs.dq, ldr = dq + 8;
    uint16_t* sQ = reinterpret_cast<uint16_t*>(xsm);
    uint16_t* sR = sQ + kMaxQ * ldr;
    uint16_t* sT = sR + 2 * kXRows * ldr;
    const int r0 = cu[s], L = cu[s + 1] - r0;
    float* Ps = P + (size_t)nq * r0;
    xattn_stage_q(sQ, ldr, hs.q, nq, dq);
    // scores S[j, q] = Q_q . k_j / sqrt(dq) into Ps
    xattn_scores(sQ, nullptr, ldr, sR, kbuf, ldkv, r0, L, nq, dq, rsqrtf((float)dq), Ps);
    // softmax over the keys of each query, in place
    const float m = xattn_reduce_q<true>(Ps, nullptr, L, nq, red);
    {
        const int q = threadIdx.x & 31, part = threadIdx.x >> 5;
        float sum = 0.f;
        if (q < nq)
            for (int j = part; j < L; j += 8) {
                const float e = expf(Ps[(size_t)j * nq + q] - m);
                Ps[(size_t)j * nq + q] = e;
                sum += e;
            }
        red[part * 32 + q] = sum;
        __syncthreads();
        float tot = 0.f;
        for (int p = 0; p < 8; ++p) tot += red[p * 32 + q];
        const float inv = 1.0f / tot;
        if (q < nq)
            for (int j = part; j < L; j += 8) Ps[(size_t)j * nq + q] *= inv;
        __syncthreads();
    }
    // O = P v, kXCols value columns at a time, keys in 32-key chunks
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    for (int c0 = 0; c0 < dq; c0 += kXCols) {
        float acc[2][4][4] = {};
        for (int j0 = 0; j0 < L; j0 += kXRows) {
            const int nr = min(kXRows, L - j0);
            __syncthreads();
            xattn_split_rows(sR, kXRows, kXCols + 8, vbuf, ldkv, (size_t)r0 + j0, nr, c0, kXCols);
            xattn_split_chunk(sT, nullptr, Ps, j0, nr, nq);
            __syncthreads();
            xattn_chunk_xr(acc, sT, sR);
        }
        // element e of tile (m, n): query 16 m + g (+ 8 for e >= 2), column
        // c0 + 32 w + 8 n + 2 t (+ 1 for odd e)
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                const int q = 16 * mt + g + 8 * hf;
                if (q >= nq) continue;
#pragma unroll
                for (int n = 0; n < 4; ++n)
                    *reinterpret_cast<float2*>(h + (size_t)s * ld_h + (size_t)q * dq + c0 +
                                               32 * warp + 8 * n + 2 * t) =
                        make_float2(acc[mt][n][2 * hf], acc[mt][n][2 * hf + 1]);
            }
    }
}

// Backward per sample: dP = dO v^T (into dS), the per-query sums
// D_q = sum_j dP P, dS = P (dP - D_q) in place, this sample's dQ
// contribution scale dS k (summed per tenant later in sample order), and,
// when kv_grads is set (the feature gradient needs them), the key rows'
// dv = P^T dO and dk = scale dS^T Q.
__global__ void __launch_bounds__(256) k_xattn_bwd(const __grid_constant__ HeadTable tab, int g0,
                                                   const int* __restrict__ cu,
                                                   const int* __restrict__ sample_slot,
                                                   int sample0, const float* __restrict__ kbuf,
                                                   const float* __restrict__ vbuf, int ldkv,
                                                   const float* __restrict__ P,
                                                   float* __restrict__ dS,
                                                   const float* __restrict__ dO, int ld_h,
                                                   float* __restrict__ dk, float* __restrict__ dv,
                                                   float* __restrict__ dQs, int kv_grads) {
    extern __shared__ __align__(16) uint8_t xsm[];
    __shared__ float red[8 * 32];
    const int s = sample0 + blockIdx.x;
    const HeadSlot& hs = tab.slot[sample_slot[s] - g0];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, dq = hs.dq, ldr = dq + 8;
    uint16_t* sQ = reinterpret_cast<uint16_t*>(xsm);
    uint16_t* sA = sQ + kMaxQ * ldr;
    uint16_t* sR = sA + 2 * kMaxQ * ldr;
    uint16_t* sT = sR + 2 * kXRows * ldr;
    uint16_t* sU = sT + 4 * kMaxQ * kXPad;
    const int r0 = cu[s], L = cu[s + 1] - r0;
    const float scale = rsqrtf((float)dq);
    const float* Ps = P + (size_t)nq * r0;
    float* dSs = dS + (size_t)nq * r0;
    xattn_stage_q(sQ, ldr, hs.q, nq, dq);
    xattn_split_rows(sA, kMaxQ, ldr, dO + (size_t)s * ld_h, dq, 0, nq, 0, dq);
    xattn_scores(sA, sA + kMaxQ * ldr, ldr, sR, vbuf, ldkv, r0, L, nq, dq, 1.f, dSs);  // dP
    const float Dq = xattn_reduce_q<false>(dSs, Ps, L, nq, red);
    {
        const int q = threadIdx.x & 31, part = threadIdx.x >> 5;
        if (q < nq)
            for (int j = part; j < L; j += 8) {
                const size_t at = (size_t)j * nq + q;
                dSs[at] = Ps[at] * (dSs[at] - Dq);
            }
        __syncthreads();
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
    const int kr = (lane & 7) + ((lane >> 3) & 1) * 8, acol = (lane >> 4) * 8;
    // sT: dS query-major (hi, lo); sU: P key-major (hi, lo), then dS key-major (hi, lo)
    uint16_t* uP = sU;
    uint16_t* uD = sU + 2 * kXRows * kXPad;
    for (int c0 = 0; c0 < dq; c0 += kXCols) {
        float aq[2][4][4] = {};
        for (int j0 = 0; j0 < L; j0 += kXRows) {
            const int nr = min(kXRows, L - j0);
            __syncthreads();
            xattn_split_rows(sR, kXRows, kXCols + 8, kbuf, ldkv, (size_t)r0 + j0, nr, c0, kXCols);
            xattn_split_chunk(sT, kv_grads ? uD : nullptr, dSs, j0, nr, nq);
            if (kv_grads) xattn_split_chunk(nullptr, uP, Ps, j0, nr, nq);
            __syncthreads();
            xattn_chunk_xr(aq, sT, sR);  // dQ += dS k
            if (!kv_grads) continue;
            // dv[j, c] = sum_q P[q, j] dO[q, c], dk[j, c] = scale sum_q dS[q, j] Q[q, c]:
            // key tiles m of the chunk, columns c0 + 32 w + 8 n, queries as the depth
            float av[2][4][4] = {}, ak[2][4][4] = {};
#pragma unroll
            for (int k0 = 0; k0 < kMaxQ; k0 += 16) {
                uint32_t ph[2][4], pl[2][4], dh[2][4], dl[2][4];
#pragma unroll
                for (int m = 0; m < 2; ++m) {
                    const size_t o = (size_t)(16 * m + kr) * kXPad + k0 + acol;
                    ldsm_x4(smem_u32(uP + o), ph[m][0], ph[m][1], ph[m][2], ph[m][3]);
                    ldsm_x4(smem_u32(uP + kXRows * kXPad + o), pl[m][0], pl[m][1], pl[m][2],
                            pl[m][3]);
                    ldsm_x4(smem_u32(uD + o), dh[m][0], dh[m][1], dh[m][2], dh[m][3]);
                    ldsm_x4(smem_u32(uD + kXRows * kXPad + o), dl[m][0], dl[m][1], dl[m][2],
                            dl[m][3]);
                }
#pragma unroll
                for (int hf = 0; hf < 2; ++hf) {
                    const size_t o = (size_t)(k0 + kr) * ldr + c0 + 32 * warp + 16 * hf + acol;
                    uint32_t oh[4], ol[4], qb[4];
                    ldsm_x4_t(smem_u32(sA + o), oh[0], oh[1], oh[2], oh[3]);
                    ldsm_x4_t(smem_u32(sA + (size_t)kMaxQ * ldr + o), ol[0], ol[1], ol[2], ol[3]);
                    ldsm_x4_t(smem_u32(sQ + o), qb[0], qb[1], qb[2], qb[3]);
#pragma unroll
                    for (int m = 0; m < 2; ++m)
#pragma unroll
                        for (int n = 0; n < 2; ++n) {
                            float(&v)[4] = av[m][2 * hf + n];
                            mma_bf16(v, ph[m][0], ph[m][1], ph[m][2], ph[m][3], oh[2 * n], oh[2 * n + 1]);
                            mma_bf16(v, ph[m][0], ph[m][1], ph[m][2], ph[m][3], ol[2 * n], ol[2 * n + 1]);
                            mma_bf16(v, pl[m][0], pl[m][1], pl[m][2], pl[m][3], oh[2 * n], oh[2 * n + 1]);
                            float(&k)[4] = ak[m][2 * hf + n];
                            mma_bf16(k, dh[m][0], dh[m][1], dh[m][2], dh[m][3], qb[2 * n], qb[2 * n + 1]);
                            mma_bf16(k, dl[m][0], dl[m][1], dl[m][2], dl[m][3], qb[2 * n], qb[2 * n + 1]);
                        }
                }
            }
            // element e of tile (m, n): key j0 + 16 m + g (+ 8 for e >= 2),
            // column c0 + 32 w + 8 n + 2 t (+ 1 for odd e)
#pragma unroll
            for (int m = 0; m < 2; ++m)
#pragma unroll
                for (int hf = 0; hf < 2; ++hf) {
                    const int j = 16 * m + g + 8 * hf;
                    if (j >= nr) continue;
                    const size_t row = (size_t)(r0 + j0 + j) * ldkv + c0 + 32 * warp + 2 * t;
#pragma unroll
                    for (int n = 0; n < 4; ++n) {
                        *reinterpret_cast<float2*>(dv + row + 8 * n) =
                            make_float2(av[m][n][2 * hf], av[m][n][2 * hf + 1]);
                        *reinterpret_cast<float2*>(dk + row + 8 * n) =
                            make_float2(ak[m][n][2 * hf] * scale, ak[m][n][2 * hf + 1] * scale);
                    }
                }
        }
#pragma unroll
        for (int mt = 0; mt < 2; ++mt)
#pragma unroll
            for (int hf = 0; hf < 2; ++hf) {
                const int q = 16 * mt + g + 8 * hf;
                if (q >= nq) continue;
#pragma unroll
                for (int n = 0; n < 4; ++n)
                    *reinterpret_cast<float2*>(dQs + (size_t)s * ld_h + (size_t)q * dq + c0 +
                                               32 * warp + 8 * n + 2 * t) =
                        make_float2(aq[mt][n][2 * hf] * scale, aq[mt][n][2 * hf + 1] * scale);
            }
    }
}

// dQ_t = sum over the slot's samples (in order) of their contributions.
template <class OT>
__global__ void __launch_bounds__(256) k_xattn_dq(const __grid_constant__ HeadTable tab,
                                                  const __grid_constant__ OT opt, AdamHp hp,
                                                  const float* __restrict__ dQs, int ld_h) {
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int i = blockIdx.y * 256 + threadIdx.x;
    if (i >= hs.nq * hs.dq) return;
    float acc = 0.f;
    for (int s = hs.s0; s < hs.s1; ++s) acc += dQs[(size_t)s * ld_h + i];
    const float g = hs.accum ? hs.g_q[i] + acc : acc;
    if constexpr (kFused<OT>)
        opt_step1(opt.slot[blockIdx.x], 4, i, g, hp);
    else
        hs.g_q[i] = g;
}

// Query-head weight gradients, re-associated through the queries.  Per
// sample, dk = scale dS^T Q and dv = P^T dO have rank <= nq (P, dS: [L, nq]
// key-major), so
//   dWk = sum_rows dk^T X = scale Q^T (sum_s G_s),  G_s = dS_s^T X_s  [nq, d]
//   dWv = sum_rows dv^T X = sum_s dO_s^T H_s,       H_s = P_s^T X_s   [nq, d]
// which takes 2 nq d flops per row and product instead of 2 dq d.  Both
// steps run in fp32 on CUDA cores (X is exact in bf16), every sum in a fixed
// order, so a tenant's gradients do not depend on the batch around it.
//
// k_xattn_gh: one CTA per (sample, 128 columns e of X), on the bf16 tensor
// cores (mma.sync m16n8k16, fp32 accumulation).  X is bf16 already; P and dS
// are fp32 and enter as two bf16 operands each, hi = bf16(P) and lo =
// bf16(P - hi), so P X = hi X + lo X to about 2^-17 of P, i.e. within the
// fp32 path's accuracy for these sums.  The sample's rows are staged 32 keys
// at a time by cp.async (X rows into padded rows; the P / dS rows, nq
// floats each, contiguous per sample), then split and transposed into
// [query][key] operands in shared memory by all threads.  Warp w computes
// columns e0 + 16 w .. + 15 (two 8-column tiles) for all 32 query rows (two
// 16-row tiles; rows past nq are zero) of both products.  The key order of
// the sums is fixed, so a sample's result does not depend on the group.
constexpr int kGhRows = 32;       // keys per staged chunk
constexpr int kGhXPad = 136;      // X row stride (bf16): conflict-free ldmatrix
constexpr int kGhAPad = 40;       // [query][key] operand row stride (bf16)

__global__ void __launch_bounds__(256) k_xattn_gh(const __grid_constant__ HeadTable tab, int g0,
                                                  const int* __restrict__ cu,
                                                  const int* __restrict__ sample_slot,
                                                  int sample0, const float* __restrict__ P,
                                                  const float* __restrict__ dS,
                                                  const uint16_t* __restrict__ X, int ldx,
                                                  float* __restrict__ Gs, float* __restrict__ Hs,
                                                  int ldg) {
    static_assert(kMaxQ == 32, "two 16-row query tiles");
    __shared__ __align__(16) uint16_t sx[2][kGhRows][kGhXPad];
    __shared__ __align__(16) float sp[2][kGhRows * kMaxQ], sd[2][kGhRows * kMaxQ];
    // split operands: [P hi, P lo, dS hi, dS lo][query][key]
    __shared__ __align__(16) uint16_t sa[4][kMaxQ][kGhAPad];
    const int s = sample0 + blockIdx.x;
    const HeadSlot& hs = tab.slot[sample_slot[s] - g0];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, e0 = blockIdx.y * 128;
    if (e0 >= hs.d_in) return;
    const int r0 = cu[s], L = cu[s + 1] - r0;
    const float* Ps = P + (size_t)nq * r0;
    const float* Ds = dS + (size_t)nq * r0;
    auto load = [&](int j0, int buf) {
        const int nr = min(kGhRows, L - j0);
        for (int i = threadIdx.x; i < kGhRows * 16; i += 256) {
            const int r = i >> 4, u = i & 15;
            const bool ok = r < nr;
            cp_async16(smem_u32(&sx[buf][r][8 * u]),
                       ok ? (const void*)(X + (size_t)(r0 + j0 + r) * ldx + e0 + 8 * u)
                          : (const void*)X,
                       ok);
        }
        const int units = nr * nq / 4;  // nr rows of nq floats, contiguous
        for (int i = threadIdx.x; i < kGhRows * kMaxQ / 4; i += 256) {
            const bool ok = i < units;
            cp_async16(smem_u32(&sp[buf][4 * i]), ok ? (const void*)(Ps + (size_t)j0 * nq + 4 * i)
                                                     : (const void*)Ps, ok);
            cp_async16(smem_u32(&sd[buf][4 * i]), ok ? (const void*)(Ds + (size_t)j0 * nq + 4 * i)
                                                     : (const void*)Ds, ok);
        }
    };
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    // acc[product: 0 = H (P), 1 = G (dS)][query tile][column tile][4]
    float acc[2][2][2][4];
#pragma unroll
    for (int a = 0; a < 2; ++a)
#pragma unroll
        for (int m = 0; m < 2; ++m)
#pragma unroll
            for (int n = 0; n < 2; ++n)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[a][m][n][e] = 0.f;
    const int nchunks = (L + kGhRows - 1) / kGhRows;
    if (nchunks > 0) load(0, 0);
    cp_async_commit();
    for (int c = 0; c < nchunks; ++c) {
        const int buf = c & 1;
        if (c + 1 < nchunks) load((c + 1) * kGhRows, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        // split and transpose: key j, query q of this chunk (rows past the
        // sample's keys or queries past nq are zero); 4 elements a thread
        const int nr = min(kGhRows, L - c * kGhRows);
        for (int i = threadIdx.x; i < kGhRows * kMaxQ; i += 256) {
            const int q = i >> 5, j = i & 31;
            const bool ok = j < nr && q < nq;
            const float pv = ok ? sp[buf][j * nq + q] : 0.f;
            const float dv = ok ? sd[buf][j * nq + q] : 0.f;
            const uint16_t ph = f2bf(pv), dh = f2bf(dv);
            sa[0][q][j] = ph;
            sa[1][q][j] = f2bf(pv - bf2f(ph));
            sa[2][q][j] = dh;
            sa[3][q][j] = f2bf(dv - bf2f(dh));
        }
        __syncthreads();
#pragma unroll
        for (int k0 = 0; k0 < kGhRows; k0 += 16) {
            // B: X rows k0..k0+15, this warp's 16 columns (two 8-column tiles)
            uint32_t b[4];
            {
                const int kr = k0 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int col = 16 * w + (lane >> 4) * 8;
                ldsm_x4_t(smem_u32(&sx[buf][kr][col]), b[0], b[1], b[2], b[3]);
            }
#pragma unroll
            for (int op = 0; op < 4; ++op) {  // P hi, P lo, dS hi, dS lo
#pragma unroll
                for (int m = 0; m < 2; ++m) {
                    uint32_t a[4];
                    const int qr = 16 * m + (lane & 7) + ((lane >> 3) & 1) * 8;
                    const int kc = k0 + (lane >> 4) * 8;
                    ldsm_x4(smem_u32(&sa[op][qr][kc]), a[0], a[1], a[2], a[3]);
                    mma_bf16(acc[op >> 1][m][0], a[0], a[1], a[2], a[3], b[0], b[1]);
                    mma_bf16(acc[op >> 1][m][1], a[0], a[1], a[2], a[3], b[2], b[3]);
                }
            }
        }
        __syncthreads();
    }
    // accumulator element e of tile (m, n): query 16 m + lane / 4 (+ 8 for
    // e >= 2), column 16 w + 8 n + 2 (lane % 4) (+ 1 for odd e)
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int q = 16 * m + (lane >> 2) + 8 * half;
            if (q >= nq) continue;
#pragma unroll
            for (int n = 0; n < 2; ++n) {
                const size_t o = ((size_t)s * kMaxQ + q) * ldg + e0 + 16 * w + 8 * n + 2 * (lane & 3);
                *reinterpret_cast<float2*>(Hs + o) =
                    make_float2(acc[0][m][n][2 * half], acc[0][m][n][2 * half + 1]);
                *reinterpret_cast<float2*>(Gs + o) =
                    make_float2(acc[1][m][n][2 * half], acc[1][m][n][2 * half + 1]);
            }
        }
}

// k_xattn_wgrad: one CTA per (slot, 32 value columns c, 64 columns e); warp
// w takes c = c0 + 4w..4w+3 (and the running sum of G_s over rows
// q = 4w..4w+3), a lane two consecutive columns e.  The slot's samples in
// order: dWv += dO_s^T H_s with dO_s [nq, 32] and H_s [nq, 64] staged; at the
// end dWk = scale Q^T G_t with G_t staged.
template <class OT>
__global__ void __launch_bounds__(256) k_xattn_wgrad(const __grid_constant__ HeadTable tab,
                                                     const __grid_constant__ OT opt, AdamHp hp,
                                                     const float* __restrict__ Gs,
                                                     const float* __restrict__ Hs, int ldg,
                                                     const float* __restrict__ dO, int ld_h) {
    __shared__ __align__(16) float sh[kMaxQ][64];
    __shared__ __align__(16) float so[kMaxQ][32];
    __shared__ __align__(16) float sg[kMaxQ][64];
    const HeadSlot& hs = tab.slot[blockIdx.x];
    if (hs.kind != JNX_HEAD_XATTN) return;
    const int nq = hs.nq, dq = hs.dq, c0 = blockIdx.y * 32, e0 = blockIdx.z * 64;
    if (c0 >= dq || e0 >= hs.d_in) return;
    const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float av[4][2], gt[4][2];
#pragma unroll
    for (int i = 0; i < 4; ++i) av[i][0] = av[i][1] = gt[i][0] = gt[i][1] = 0.f;
    for (int s = hs.s0; s < hs.s1; ++s) {
        __syncthreads();  // the previous sample's staged rows are read
        for (int i = threadIdx.x; i < nq * 16; i += 256) {  // H_s [nq, 64]: 16 float4 per row
            const int q = i >> 4, u = i & 15;
            *reinterpret_cast<float4*>(&sh[q][4 * u]) = *reinterpret_cast<const float4*>(
                Hs + ((size_t)s * kMaxQ + q) * ldg + e0 + 4 * u);
        }
        for (int i = threadIdx.x; i < nq * 8; i += 256) {  // dO_s [nq, 32]: 8 float4 per row
            const int q = i >> 3, u = i & 7;
            *reinterpret_cast<float4*>(&so[q][4 * u]) = *reinterpret_cast<const float4*>(
                dO + (size_t)s * ld_h + (size_t)q * dq + c0 + 4 * u);
        }
        if (4 * w < nq) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float2 gv = *reinterpret_cast<const float2*>(
                    Gs + ((size_t)s * kMaxQ + 4 * w + i) * ldg + e0 + 2 * lane);
                gt[i][0] += gv.x;
                gt[i][1] += gv.y;
            }
        }
        __syncthreads();
        for (int q = 0; q < nq; ++q) {
            const float4 o4 = *reinterpret_cast<const float4*>(&so[q][4 * w]);
            const float2 hv = *reinterpret_cast<const float2*>(&sh[q][2 * lane]);
            const float o[4] = {o4.x, o4.y, o4.z, o4.w};
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                av[i][0] = fmaf(o[i], hv.x, av[i][0]);
                av[i][1] = fmaf(o[i], hv.y, av[i][1]);
            }
        }
    }
    __syncthreads();
    if (4 * w < nq) {
#pragma unroll
        for (int i = 0; i < 4; ++i)
            *reinterpret_cast<float2*>(&sg[4 * w + i][2 * lane]) = make_float2(gt[i][0], gt[i][1]);
    }
    __syncthreads();
    const float scale = rsqrtf((float)dq);
    float ak[4][2] = {};
    for (int q = 0; q < nq; ++q) {
        const float2 gv = *reinterpret_cast<const float2*>(&sg[q][2 * lane]);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float qv = bf2f(hs.q[(size_t)q * dq + c0 + 4 * w + i]);
            ak[i][0] = fmaf(qv, gv.x, ak[i][0]);
            ak[i][1] = fmaf(qv, gv.y, ak[i][1]);
        }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const size_t o = (size_t)(c0 + 4 * w + i) * hs.d_in + e0 + 2 * lane;
        float2 vk = make_float2(ak[i][0] * scale, ak[i][1] * scale);
        float2 vv = make_float2(av[i][0], av[i][1]);
        if (hs.accum) {
            const float2 ok = *reinterpret_cast<const float2*>(hs.g_wk + o);
            const float2 ov = *reinterpret_cast<const float2*>(hs.g_wv + o);
            vk.x += ok.x;
            vk.y += ok.y;
            vv.x += ov.x;
            vv.y += ov.y;
        }
        if constexpr (kFused<OT>) {
            opt_step2(opt.slot[blockIdx.x], 5, o, vk, hp);
            opt_step2(opt.slot[blockIdx.x], 6, o, vv, hp);
        } else {
            *reinterpret_cast<float2*>(hs.g_wk + o) = vk;
            *reinterpret_cast<float2*>(hs.g_wv + o) = vv;
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
        k_head_lin<1><<<dim3((b.max_ns + kLinS - 1) / kLinS,
                             (b.max_mlp_hid + kLinCols - 1) / kLinCols, b.n),
                        256, kLinSmem, s>>>(
            tab, pooled, d, ws.z, ws.h, ws.ld_h, sample_target, preds);
    if (b.any_xattn) {
        const size_t smem = xattn_smem_bytes(b.max_dq, false);
        k_xattn_fwd<<<b.sample1 - b.sample0, 256, smem, s>>>(tab, b.g0, cu, sample_slot,
                                                             b.sample0, ws.kbuf, ws.vbuf, ws.ldkv,
                                                             ws.P, ws.h, ws.ld_h);
    }
    k_head_lin<2><<<dim3((b.max_ns + kLinS - 1) / kLinS,
                         (b.max_width + kLinCols - 1) / kLinCols, b.n),
                    256, kLinSmem, s>>>(
        tab, ws.h, ws.ld_h, ws.y, nullptr, ws.ld_y, sample_target, preds);
    if (targets)  // without targets (inference) there is no loss
        k_l2_loss<<<b.n, 256, 0, s>>>(tab, ws.y, ws.ld_y, targets, sample_target, ws.dy, loss);
    return cuda_ok("heads forward");
}

jnx_status heads_backward_launch(const HeadTable& tab, const HeadBatch& b, const HeadScratch& ws,
                                 const float* pooled, int d, const uint16_t* hidden,
                                 const int* cu, const int* sample_slot, bool kv_grads,
                                 cudaStream_t s) {
    if (b.n == 0) return JNX_OK;
    const NoOpt no{};
    const AdamHp nh{};
    k_head_dw_out<NoOpt>
        <<<dim3(b.n, (b.max_width + 15) / 16, (b.max_hid + 255) / 256), 256, 0, s>>>(
            tab, no, nh, ws.dy, ws.ld_y, ws.h, ws.ld_h);
    k_head_back_in<<<dim3(b.n, (b.max_hid + 1023) / 1024, (b.max_ns + 7) / 8), 256, 0, s>>>(
        tab, ws.dy, ws.ld_y, ws.z, ws.ld_h, ws.dh);
    if (b.any_mlp)
        k_mlp_dw1<NoOpt><<<dim3(b.n, (b.max_mlp_hid + kDw1Rows - 1) / kDw1Rows, (d / 4 + 255) / 256),
                           256, 0, s>>>(
            tab, no, nh, ws.dh, ws.ld_h, pooled, d);
    if (b.any_xattn) {
        const size_t smem = xattn_smem_bytes(b.max_dq, true);
        k_xattn_bwd<<<b.sample1 - b.sample0, 256, smem, s>>>(
            tab, b.g0, cu, sample_slot, b.sample0, ws.kbuf, ws.vbuf, ws.ldkv, ws.P, ws.dS, ws.dh,
            ws.ld_h, ws.dk, ws.dv, ws.dQs, kv_grads ? 1 : 0);
        k_xattn_dq<NoOpt><<<dim3(b.n, (b.max_nq * b.max_dq + 255) / 256), 256, 0, s>>>(
            tab, no, nh, ws.dQs, ws.ld_h);
        k_xattn_gh<<<dim3(b.sample1 - b.sample0, d / 128), 256, 0, s>>>(
            tab, b.g0, cu, sample_slot, b.sample0, ws.P, ws.dS, hidden, d, ws.Gs, ws.Hs, d);
        k_xattn_wgrad<NoOpt><<<dim3(b.n, b.max_dq / 32, d / 64), 256, 0, s>>>(
            tab, no, nh, ws.Gs, ws.Hs, d, ws.dh, ws.ld_h);
    }
    return cuda_ok("heads backward");
}

jnx_status heads_backward_front_launch(const HeadTable& tab, const HeadBatch& b,
                                       const HeadScratch& ws, int d, const uint16_t* hidden,
                                       const int* cu, const int* sample_slot, bool kv_grads,
                                       cudaStream_t s) {
    if (b.n == 0) return JNX_OK;
    k_head_back_in<<<dim3(b.n, (b.max_hid + 1023) / 1024, (b.max_ns + 7) / 8), 256, 0, s>>>(
        tab, ws.dy, ws.ld_y, ws.z, ws.ld_h, ws.dh);
    if (b.any_xattn) {
        const size_t smem = xattn_smem_bytes(b.max_dq, true);
        k_xattn_bwd<<<b.sample1 - b.sample0, 256, smem, s>>>(
            tab, b.g0, cu, sample_slot, b.sample0, ws.kbuf, ws.vbuf, ws.ldkv, ws.P, ws.dS, ws.dh,
            ws.ld_h, ws.dk, ws.dv, ws.dQs, kv_grads ? 1 : 0);
        k_xattn_gh<<<dim3(b.sample1 - b.sample0, d / 128), 256, 0, s>>>(
            tab, b.g0, cu, sample_slot, b.sample0, ws.P, ws.dS, hidden, d, ws.Gs, ws.Hs, d);
    }
    return cuda_ok("heads backward");
}

jnx_status heads_backward_step_launch(const HeadTable& tab, const HeadOptTable& opt,
                                      const AdamHp& hp, const HeadBatch& b,
                                      const HeadScratch& ws, const float* pooled, int d,
                                      cudaStream_t s) {
    if (b.n == 0) return JNX_OK;
    k_head_dw_out<HeadOptTable>
        <<<dim3(b.n, (b.max_width + 15) / 16, (b.max_hid + 255) / 256), 256, 0, s>>>(
            tab, opt, hp, ws.dy, ws.ld_y, ws.h, ws.ld_h);
    if (b.any_mlp)
        k_mlp_dw1<HeadOptTable>
            <<<dim3(b.n, (b.max_mlp_hid + kDw1Rows - 1) / kDw1Rows, (d / 4 + 255) / 256), 256, 0,
               s>>>(
            tab, opt, hp, ws.dh, ws.ld_h, pooled, d);
    if (b.any_xattn) {
        // wgrad reads the learned queries, which dq then updates
        k_xattn_wgrad<HeadOptTable><<<dim3(b.n, b.max_dq / 32, d / 64), 256, 0, s>>>(
            tab, opt, hp, ws.Gs, ws.Hs, d, ws.dh, ws.ld_h);
        k_xattn_dq<HeadOptTable><<<dim3(b.n, (b.max_nq * b.max_dq + 255) / 256), 256, 0, s>>>(
            tab, opt, hp, ws.dQs, ws.ld_h);
    }
    return cuda_ok("heads backward step");
}

jnx_status heads_set_smem() {
    static std::atomic<uint64_t> fwd{0}, bwd{0}, lin1{0}, lin2{0};
    if (set_smem_limit(reinterpret_cast<const void*>(k_xattn_fwd),
                       (int)xattn_smem_bytes(512, false), fwd) != cudaSuccess ||
        set_smem_limit(reinterpret_cast<const void*>(k_xattn_bwd),
                       (int)xattn_smem_bytes(512, true), bwd) != cudaSuccess ||
        set_smem_limit(reinterpret_cast<const void*>(k_head_lin<1>), kLinSmem, lin1) !=
            cudaSuccess ||
        set_smem_limit(reinterpret_cast<const void*>(k_head_lin<2>), kLinSmem, lin2) !=
            cudaSuccess)
        return cuda_ok("heads smem attribute");
    return JNX_OK;
}

}  // namespace jnx
