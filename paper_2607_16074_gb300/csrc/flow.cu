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
// runs on bf16 mma.sync tiles with fp32 softmax; the small per-row and
// per-sample pieces run on CUDA cores in fp32.
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
// time embedding: s(tau), z1 = T1 s + tb1, phi = T2 SiLU(z1) + tb2.  Each
// layer is one launch over (sample, block of 32 output rows): one warp per
// row, lanes along the dot product with 16-byte weight loads (dm is a
// multiple of 256), the row sum in a fixed butterfly order.
// ---------------------------------------------------------------------------
constexpr int kTimeRows = 32;

// dot product of the bf16 row w [dm] with the fp32 vector v [dm] in shared
// memory, summed over the warp (every lane returns the sum)
__device__ __forceinline__ float warp_row_dot(const uint16_t* __restrict__ w,
                                              const float* __restrict__ v, int dm, int lane) {
    float acc = 0.f;
    for (int k = 8 * lane; k < dm; k += 256) {
        const uint4 q = *reinterpret_cast<const uint4*>(w + k);
        const uint32_t u[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            acc = fmaf(__uint_as_float(u[e] << 16), v[k + 2 * e], acc);
            acc = fmaf(__uint_as_float(u[e] & 0xffff0000u), v[k + 2 * e + 1], acc);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

__global__ void __launch_bounds__(256) k_flow_time1(const float* __restrict__ tau,
                                                    const int* __restrict__ sample_slot,
                                                    const __grid_constant__ FlowSlots fs,
                                                    FlowDims dd, const uint16_t* __restrict__ t1,
                                                    const uint16_t* __restrict__ tb1,
                                                    float* __restrict__ sfeat,
                                                    float* __restrict__ z1) {
    extern __shared__ float sh[];  // s(tau) [dm]
    const int s = blockIdx.x, dm = dd.dm, half = dm / 2;
    const int t = fs.tenant[sample_slot[s]];
    const float tv = tau[s];
    for (int i = threadIdx.x; i < dm; i += blockDim.x) {
        const int k = i < half ? i : i - half;
        const float w = powf(10000.f, -(float)k / (float)half);
        const float a = 1000.f * tv * w;
        const float v = i < half ? sinf(a) : cosf(a);
        sh[i] = v;
        if (blockIdx.y == 0) sfeat[(size_t)s * dm + i] = v;
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint16_t* T1 = t1 + (size_t)t * dm * dm;
    for (int j = blockIdx.y * kTimeRows + warp; j < (blockIdx.y + 1) * kTimeRows; j += 8) {
        const float acc = warp_row_dot(T1 + (size_t)j * dm, sh, dm, lane);
        if (lane == 0) z1[(size_t)s * dm + j] = acc + bf2f(tb1[(size_t)t * dm + j]);
    }
}

__global__ void __launch_bounds__(256) k_flow_time2(const int* __restrict__ sample_slot,
                                                    const __grid_constant__ FlowSlots fs,
                                                    FlowDims dd, const uint16_t* __restrict__ t2,
                                                    const uint16_t* __restrict__ tb2,
                                                    const float* __restrict__ z1,
                                                    float* __restrict__ phi) {
    extern __shared__ float sh[];  // SiLU(z1) [dm]
    const int s = blockIdx.x, dm = dd.dm;
    const int t = fs.tenant[sample_slot[s]];
    for (int i = threadIdx.x; i < dm; i += blockDim.x) sh[i] = silu_f(z1[(size_t)s * dm + i]);
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint16_t* T2 = t2 + (size_t)t * dm * dm;
    for (int j = blockIdx.y * kTimeRows + warp; j < (blockIdx.y + 1) * kTimeRows; j += 8) {
        const float acc = warp_row_dot(T2 + (size_t)j * dm, sh, dm, lane);
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
// attention on the warp-level bf16 tensor-core path (mma.sync m16n8k16, fp32
// accumulation).  Per (sample, head): the C action queries against the
// sample's L context keys then its C action keys, bidirectional.  Keys are
// staged 64 at a time by cp.async into shared-memory rows of 64 bf16 (128
// bytes, the 16-byte units XOR-swizzled by the row's low three bits, so the
// ldmatrix row gathers hit distinct banks).  Query rows past C are zero and
// never stored; key rows past L + C are zero and masked.
//   qkv [M_a, 3 dm] bf16 (q | k_a | v_a), kvc [N, 2 dm] bf16 (k_c | v_c),
//   o [M_a, dm] bf16, lse [M_a, nh] fp32: the log2 of the softmax
//   denominator of the log2e-scaled scores, their maximum included.
// ---------------------------------------------------------------------------
constexpr int kKT = 64;          // keys per staged tile
constexpr int kRowB = kHd * 2;   // bytes per staged row
constexpr int kTileB = kKT * kRowB;

__device__ __forceinline__ uint32_t swz(int row, int unit) {
    return (uint32_t)(row * kRowB + ((unit ^ (row & 7)) << 4));
}

// Key j of the sample (context rows first, then its action rows): its K row;
// the V row follows dm elements later in both buffers.
__device__ __forceinline__ const uint16_t* key_row(int j, int L, const uint16_t* kvc, int ctx0,
                                                   const uint16_t* qkv, int act0, int dm, int h) {
    return j < L ? kvc + (size_t)(ctx0 + j) * 2 * dm + h * kHd
                 : qkv + (size_t)(act0 + j - L) * 3 * dm + dm + h * kHd;
}

// cp.async of keys j0 .. j0 + 63 into the K tile at sk and the V tile at sv.
__device__ __forceinline__ void load_kv_tile(uint32_t sk, uint32_t sv, int j0, int nkeys, int L,
                                             const uint16_t* kvc, int ctx0, const uint16_t* qkv,
                                             int act0, int dm, int h) {
    for (int i = threadIdx.x; i < kKT * 8; i += blockDim.x) {
        const int r = i >> 3, u = i & 7, j = j0 + r;
        const bool ok = j < nkeys;
        const uint16_t* kr = ok ? key_row(j, L, kvc, ctx0, qkv, act0, dm, h) : qkv;
        cp_async16(sk + swz(r, u), kr + 8 * u, ok);
        cp_async16(sv + swz(r, u), kr + dm + 8 * u, ok);
    }
}

// cp.async of the bf16 rows 0 .. C - 1 (row stride ld) into a tile of `rows`
// rows at dst; rows C .. rows - 1 zero.
__device__ __forceinline__ void load_rows(uint32_t dst, const uint16_t* src, size_t ld, int C,
                                          int rows) {
    for (int i = threadIdx.x; i < rows * 8; i += blockDim.x) {
        const int r = i >> 3, u = i & 7;
        const bool ok = r < C;
        cp_async16(dst + swz(r, u), ok ? src + (size_t)r * ld + 8 * u : src, ok);
    }
}

// The fp32 rows 0 .. C - 1 (row stride ld) as bf16 into a tile of `rows` rows
// at dst (generic pointer); rows C .. rows - 1 zero.
__device__ __forceinline__ void store_rows_bf16(uint8_t* dst, const float* src, size_t ld, int C,
                                                int rows) {
    for (int i = threadIdx.x; i < rows * 8; i += blockDim.x) {
        const int r = i >> 3, u = i & 7;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r < C) {
            const float4 a = *reinterpret_cast<const float4*>(src + (size_t)r * ld + 8 * u);
            const float4 b = *reinterpret_cast<const float4*>(src + (size_t)r * ld + 8 * u + 4);
            v = make_uint4(pack_bf2(a.x, a.y), pack_bf2(a.z, a.w), pack_bf2(b.x, b.y),
                           pack_bf2(b.z, b.w));
        }
        *reinterpret_cast<uint4*>(dst + swz(r, u)) = v;
    }
}

// A operand (16 rows from row0, k16 step kk) from a swizzled row tile.
__device__ __forceinline__ void ld_a(uint32_t base, int row0, int kk, int lane, uint32_t (&a)[4]) {
    const int mi = lane >> 3, rr = lane & 7;
    ldsm_x4(base + swz(row0 + rr + 8 * (mi & 1), kk * 2 + (mi >> 1)), a[0], a[1], a[2], a[3]);
}
// B operand of two n8 tiles (rows n0 .. n0 + 15 hold n, their columns k;
// k16 step kk): b0, b1 for the first tile, b2, b3 for the second.
__device__ __forceinline__ void ld_b(uint32_t base, int n0, int kk, int lane, uint32_t (&b)[4]) {
    const int mi = lane >> 3, rr = lane & 7;
    ldsm_x4(base + swz(n0 + rr + 8 * (mi >> 1), kk * 2 + (mi & 1)), b[0], b[1], b[2], b[3]);
}
// B operand of two n8 tiles (columns 16 dn .. 16 dn + 15 hold n, rows
// k0 .. k0 + 15 hold k).
__device__ __forceinline__ void ld_bt(uint32_t base, int k0, int dn, int lane, uint32_t (&b)[4]) {
    const int mi = lane >> 3, rr = lane & 7;
    ldsm_x4_t(base + swz(k0 + rr + 8 * (mi & 1), dn * 2 + (mi >> 1)), b[0], b[1], b[2], b[3]);
}
// Two n8 accumulator tiles (16 rows x 16 columns) as the bf16 A operand of
// the next product (its k = their columns).
__device__ __forceinline__ void acc_to_a(const float (&c0)[4], const float (&c1)[4],
                                         uint32_t (&a)[4]) {
    a[0] = pack_bf2(c0[0], c0[1]);
    a[1] = pack_bf2(c0[2], c0[3]);
    a[2] = pack_bf2(c1[0], c1[1]);
    a[3] = pack_bf2(c1[2], c1[3]);
}
__device__ __forceinline__ void mma4(float (&c)[4], const uint32_t (&a)[4], uint32_t b0,
                                     uint32_t b1) {
    mma_bf16(c, a[0], a[1], a[2], a[3], b0, b1);
}

// Forward.  One CTA of four warps per (sample, head); warp w takes query
// tile w / KS (16 rows) and the w % KS-th of the 64 / KS-key slices of every
// staged tile, with its own running maximum and sum; the KS slices are
// merged at the end in slice order.
template <int KS>
__global__ void __launch_bounds__(128) k_flow_attn_fwd(const uint16_t* __restrict__ qkv,
                                                       const uint16_t* __restrict__ kvc,
                                                       const int* __restrict__ cu, FlowDims dd,
                                                       uint16_t* __restrict__ o,
                                                       float* __restrict__ lse) {
    constexpr int NK = kKT / KS, NT = NK / 8;
    __shared__ __align__(128) uint8_t sbuf[4 * kTileB];  // (K, V) x 2 buffers
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
    const int MT = (C + 15) >> 4, mt = warp / KS, ks = warp % KS;
    const bool active = mt < MT;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C, nkeys = L + C;
    const uint32_t sb = smem_u32(sbuf);
    load_rows(sb, qkv + (size_t)act0 * 3 * dm + h * kHd, 3 * dm, C, MT * 16);
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();
    uint32_t qa[4][4];
    if (active)
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) ld_a(sb, mt * 16, kk, lane, qa[kk]);
    __syncthreads();
    float oacc[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) oacc[i][0] = oacc[i][1] = oacc[i][2] = oacc[i][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.f, 0.f};
    const float sc2 = kLog2e / sqrtf((float)kHd);
    const int ntiles = (nkeys + kKT - 1) / kKT;
    load_kv_tile(sb, sb + kTileB, 0, nkeys, L, kvc, ctx0, qkv, act0, dm, h);
    cp_async_commit();
    for (int t = 0; t < ntiles; ++t) {
        const uint32_t kb = sb + (t & 1) * 2 * kTileB, vb = kb + kTileB;
        if (t + 1 < ntiles) {
            const uint32_t nk = sb + ((t + 1) & 1) * 2 * kTileB;
            load_kv_tile(nk, nk + kTileB, (t + 1) * kKT, nkeys, L, kvc, ctx0, qkv, act0, dm, h);
        }
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (active) {
            float sacc[NT][4];
#pragma unroll
            for (int i = 0; i < NT; ++i) sacc[i][0] = sacc[i][1] = sacc[i][2] = sacc[i][3] = 0.f;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
#pragma unroll
                for (int nb = 0; nb < NT / 2; ++nb) {
                    uint32_t b[4];
                    ld_b(kb, ks * NK + nb * 16, kk, lane, b);
                    mma4(sacc[2 * nb], qa[kk], b[0], b[1]);
                    mma4(sacc[2 * nb + 1], qa[kk], b[2], b[3]);
                }
            float mx[2] = {mrow[0], mrow[1]};
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = t * kKT + ks * NK + nt * 8 + 2 * tq + (e & 1);
                    const float v = j < nkeys ? sacc[nt][e] * sc2 : -INFINITY;
                    sacc[nt][e] = v;
                    mx[e >> 1] = fmaxf(mx[e >> 1], v);
                }
            float alpha[2];
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 1));
                mx[i] = fmaxf(mx[i], __shfl_xor_sync(0xffffffffu, mx[i], 2));
                alpha[i] = mx[i] == -INFINITY ? 1.f : exp2f(mrow[i] - mx[i]);
                mrow[i] = mx[i];
                lrow[i] *= alpha[i];
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float m = mx[e >> 1];
                    const float p = m == -INFINITY ? 0.f : exp2f(sacc[nt][e] - m);
                    sacc[nt][e] = p;
                    lrow[e >> 1] += p;
                }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                oacc[i][0] *= alpha[0];
                oacc[i][1] *= alpha[0];
                oacc[i][2] *= alpha[1];
                oacc[i][3] *= alpha[1];
            }
#pragma unroll
            for (int k2 = 0; k2 < NK / 16; ++k2) {
                uint32_t pa[4];
                acc_to_a(sacc[2 * k2], sacc[2 * k2 + 1], pa);
#pragma unroll
                for (int dn = 0; dn < 4; ++dn) {
                    uint32_t b[4];
                    ld_bt(vb, ks * NK + k2 * 16, dn, lane, b);
                    mma4(oacc[2 * dn], pa, b[0], b[1]);
                    mma4(oacc[2 * dn + 1], pa, b[2], b[3]);
                }
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 2; ++i) {
        lrow[i] += __shfl_xor_sync(0xffffffffu, lrow[i], 1);
        lrow[i] += __shfl_xor_sync(0xffffffffu, lrow[i], 2);
    }
    if (KS == 1) {
        if (!active) return;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int c = mt * 16 + g + 8 * i;
            if (c >= C) continue;
            const float inv = 1.f / lrow[i];
            uint16_t* orow = o + (size_t)(act0 + c) * dm + h * kHd;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
                *reinterpret_cast<uint32_t*>(orow + nt * 8 + 2 * tq) =
                    pack_bf2(oacc[nt][2 * i] * inv, oacc[nt][2 * i + 1] * inv);
            if (tq == 0) lse[(size_t)(act0 + c) * dd.nh + h] = mrow[i] + log2f(lrow[i]);
        }
        return;
    }
    // merge the KS slices: per warp its 16 x 64 partial output, maximum and sum
    float* mo = reinterpret_cast<float*>(sbuf);  // [4][16][kHd + 1]
    float* mm = mo + 4 * 16 * (kHd + 1);         // [4][16]
    float* ml = mm + 4 * 16;                     // [4][16]
    if (active) {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int r = g + 8 * i;
            float* row = mo + (warp * 16 + r) * (kHd + 1);
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                row[nt * 8 + 2 * tq] = oacc[nt][2 * i];
                row[nt * 8 + 2 * tq + 1] = oacc[nt][2 * i + 1];
            }
            if (tq == 0) {
                mm[warp * 16 + r] = mrow[i];
                ml[warp * 16 + r] = lrow[i];
            }
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < MT * 16 * (kHd / 2); i += blockDim.x) {
        const int r = i / (kHd / 2), e = 2 * (i % (kHd / 2));
        if (r >= C) continue;
        const int w0 = (r >> 4) * KS, rl = r & 15;
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < KS; ++k) M = fmaxf(M, mm[(w0 + k) * 16 + rl]);
        float Ls = 0.f, v0 = 0.f, v1 = 0.f;
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            const float mk = mm[(w0 + k) * 16 + rl];
            const float wk = mk == -INFINITY ? 0.f : exp2f(mk - M);
            const float* row = mo + ((w0 + k) * 16 + rl) * (kHd + 1);
            Ls += ml[(w0 + k) * 16 + rl] * wk;
            v0 += row[e] * wk;
            v1 += row[e + 1] * wk;
        }
        const float inv = 1.f / Ls;
        *reinterpret_cast<uint32_t*>(o + (size_t)(act0 + r) * dm + h * kHd + e) =
            pack_bf2(v0 * inv, v1 * inv);
        if (e == 0) lse[(size_t)(act0 + r) * dd.nh + h] = M + log2f(Ls);
    }
}

// Query-row prologue of the backward: q (and dO as bf16) into shared tiles,
// D_c = dO_c . o_c (fp32) and the forward's lse per row; rows past C get
// D = 0, lse = +inf (so their probabilities are 0).
__device__ __forceinline__ void bwd_query_side(uint32_t sq, uint8_t* sg_gen, float* sD, float* sL,
                                               const uint16_t* qkv, const uint16_t* o,
                                               const float* dO, const float* lse, int act0, int C,
                                               int rows, int dm, int nh, int h) {
    load_rows(sq, qkv + (size_t)act0 * 3 * dm + h * kHd, 3 * dm, C, rows);
    cp_async_commit();
    store_rows_bf16(sg_gen, dO + (size_t)act0 * dm + h * kHd, dm, C, rows);
    for (int c = threadIdx.x; c < rows; c += blockDim.x) {
        float Dc = 0.f, lc = INFINITY;
        if (c < C) {
            const size_t r = (size_t)(act0 + c);
            const float* gr = dO + r * dm + h * kHd;
            const uint16_t* orow = o + r * dm + h * kHd;
            for (int e = 0; e < kHd; ++e) Dc += gr[e] * bf2f(orow[e]);
            lc = lse[r * nh + h];
        }
        sD[c] = Dc;
        sL[c] = lc;
    }
    cp_async_wait<0>();
    __syncthreads();
}

// Backward, query side: dq_c = scale sum_j dS_cj k_j, dS = P (dP - D_c),
// dP_cj = dO_c . v_j, P from the forward's lse.  Warps split as the forward
// (query tile, key slice); the KS partial dq are summed in slice order.
template <int KS>
__global__ void __launch_bounds__(128) k_flow_attn_bwd_q(
    const uint16_t* __restrict__ qkv, const uint16_t* __restrict__ kvc, const int* __restrict__ cu,
    FlowDims dd, const uint16_t* __restrict__ o, const float* __restrict__ dO,
    const float* __restrict__ lse, uint16_t* __restrict__ dqkv) {
    constexpr int NK = kKT / KS, NT = NK / 8;
    __shared__ __align__(128) uint8_t sbuf[4 * kTileB];
    __shared__ float sD[kMaxC], sL[kMaxC];
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
    const int MT = (C + 15) >> 4, mt = warp / KS, ks = warp % KS;
    const bool active = mt < MT;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C, nkeys = L + C;
    const uint32_t sb = smem_u32(sbuf);
    bwd_query_side(sb, sbuf + kTileB, sD, sL, qkv, o, dO, lse, act0, C, MT * 16, dm, dd.nh, h);
    uint32_t qa[4][4], ga[4][4];
    float lr[2] = {0.f, 0.f}, Dr[2] = {0.f, 0.f};
    if (active) {
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            ld_a(sb, mt * 16, kk, lane, qa[kk]);
            ld_a(sb + kTileB, mt * 16, kk, lane, ga[kk]);
        }
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int c = mt * 16 + g + 8 * i;
            lr[i] = c < C ? sL[c] : 0.f;
            Dr[i] = sD[c];
        }
    }
    __syncthreads();
    float dq[8][4];
#pragma unroll
    for (int i = 0; i < 8; ++i) dq[i][0] = dq[i][1] = dq[i][2] = dq[i][3] = 0.f;
    const float sc2 = kLog2e / sqrtf((float)kHd);
    const int ntiles = (nkeys + kKT - 1) / kKT;
    load_kv_tile(sb, sb + kTileB, 0, nkeys, L, kvc, ctx0, qkv, act0, dm, h);
    cp_async_commit();
    for (int t = 0; t < ntiles; ++t) {
        const uint32_t kb = sb + (t & 1) * 2 * kTileB, vb = kb + kTileB;
        if (t + 1 < ntiles) {
            const uint32_t nk = sb + ((t + 1) & 1) * 2 * kTileB;
            load_kv_tile(nk, nk + kTileB, (t + 1) * kKT, nkeys, L, kvc, ctx0, qkv, act0, dm, h);
        }
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (active) {
            float sacc[NT][4], dp[NT][4];
#pragma unroll
            for (int i = 0; i < NT; ++i)
#pragma unroll
                for (int e = 0; e < 4; ++e) sacc[i][e] = dp[i][e] = 0.f;
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
#pragma unroll
                for (int nb = 0; nb < NT / 2; ++nb) {
                    uint32_t b[4];
                    ld_b(kb, ks * NK + nb * 16, kk, lane, b);
                    mma4(sacc[2 * nb], qa[kk], b[0], b[1]);
                    mma4(sacc[2 * nb + 1], qa[kk], b[2], b[3]);
                    ld_b(vb, ks * NK + nb * 16, kk, lane, b);
                    mma4(dp[2 * nb], ga[kk], b[0], b[1]);
                    mma4(dp[2 * nb + 1], ga[kk], b[2], b[3]);
                }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt)
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int j = t * kKT + ks * NK + nt * 8 + 2 * tq + (e & 1);
                    const float p = j < nkeys ? exp2f(sacc[nt][e] * sc2 - lr[e >> 1]) : 0.f;
                    sacc[nt][e] = p * (dp[nt][e] - Dr[e >> 1]);
                }
#pragma unroll
            for (int k2 = 0; k2 < NK / 16; ++k2) {
                uint32_t da[4];
                acc_to_a(sacc[2 * k2], sacc[2 * k2 + 1], da);
#pragma unroll
                for (int dn = 0; dn < 4; ++dn) {
                    uint32_t b[4];
                    ld_bt(kb, ks * NK + k2 * 16, dn, lane, b);
                    mma4(dq[2 * dn], da, b[0], b[1]);
                    mma4(dq[2 * dn + 1], da, b[2], b[3]);
                }
            }
        }
        __syncthreads();
    }
    const float sc = 1.f / sqrtf((float)kHd);
    if (KS == 1) {
        if (!active) return;
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int c = mt * 16 + g + 8 * i;
            if (c >= C) continue;
            uint16_t* dr = dqkv + (size_t)(act0 + c) * 3 * dm + h * kHd;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
                *reinterpret_cast<uint32_t*>(dr + nt * 8 + 2 * tq) =
                    pack_bf2(dq[nt][2 * i] * sc, dq[nt][2 * i + 1] * sc);
        }
        return;
    }
    float* mo = reinterpret_cast<float*>(sbuf);  // [4][16][kHd + 1]
    if (active) {
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            float* row = mo + (warp * 16 + g + 8 * i) * (kHd + 1);
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                row[nt * 8 + 2 * tq] = dq[nt][2 * i];
                row[nt * 8 + 2 * tq + 1] = dq[nt][2 * i + 1];
            }
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < MT * 16 * (kHd / 2); i += blockDim.x) {
        const int r = i / (kHd / 2), e = 2 * (i % (kHd / 2));
        if (r >= C) continue;
        const int w0 = (r >> 4) * KS, rl = r & 15;
        float v0 = 0.f, v1 = 0.f;
#pragma unroll
        for (int k = 0; k < KS; ++k) {
            const float* row = mo + ((w0 + k) * 16 + rl) * (kHd + 1);
            v0 += row[e];
            v1 += row[e + 1];
        }
        *reinterpret_cast<uint32_t*>(dqkv + (size_t)(act0 + r) * 3 * dm + h * kHd + e) =
            pack_bf2(v0 * sc, v1 * sc);
    }
}

// Backward, key side: per key j, dv_j = sum_c P_cj dO_c and dk_j = scale
// sum_c dS_cj q_c over the NQ x 16 (padded) queries.  One CTA of four warps
// per (sample, head, key-tile stride): tiles blockIdx.z, blockIdx.z +
// gridDim.z, ...; warp w owns keys 16 w .. 16 w + 15 of each tile.  Each key's
// gradients are complete in one pass (no accumulation across CTAs).
template <int NQ>
__global__ void __launch_bounds__(128) k_flow_attn_bwd_kv(
    const uint16_t* __restrict__ qkv, const uint16_t* __restrict__ kvc, const int* __restrict__ cu,
    FlowDims dd, const uint16_t* __restrict__ o, const float* __restrict__ dO,
    const float* __restrict__ lse, uint16_t* __restrict__ dqkv, uint16_t* __restrict__ dkvc) {
    constexpr int NT = 2 * NQ;  // n8 query tiles
    __shared__ __align__(128) uint8_t sbuf[4 * kTileB];  // q, dO, K, V
    __shared__ float sD[kMaxC], sL[kMaxC];
    const int s = blockIdx.x, h = blockIdx.y, C = dd.C, dm = dd.dm;
    const int ctx0 = cu[s], L = cu[s + 1] - ctx0, act0 = s * C, nkeys = L + C;
    const int ntiles = (nkeys + kKT - 1) / kKT;
    if ((int)blockIdx.z >= ntiles) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, g = lane >> 2, tq = lane & 3;
    const uint32_t sq = smem_u32(sbuf), sg = sq + kTileB, kb = sq + 2 * kTileB, vb = kb + kTileB;
    bwd_query_side(sq, sbuf + kTileB, sD, sL, qkv, o, dO, lse, act0, C, NQ * 16, dm, dd.nh, h);
    const float sc2 = kLog2e / sqrtf((float)kHd), sc = 1.f / sqrtf((float)kHd);
    for (int t = blockIdx.z; t < ntiles; t += gridDim.z) {
        __syncthreads();  // the previous tile's readers are done
        load_kv_tile(kb, vb, t * kKT, nkeys, L, kvc, ctx0, qkv, act0, dm, h);
        cp_async_commit();
        cp_async_wait<0>();
        __syncthreads();
        const int k0 = t * kKT + warp * 16;
        if (k0 >= nkeys) continue;
        float st[NT][4], dpt[NT][4];
#pragma unroll
        for (int i = 0; i < NT; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) st[i][e] = dpt[i][e] = 0.f;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk) {
            uint32_t ka[4], va[4];
            ld_a(kb, warp * 16, kk, lane, ka);
            ld_a(vb, warp * 16, kk, lane, va);
#pragma unroll
            for (int nb = 0; nb < NQ; ++nb) {
                uint32_t b[4];
                ld_b(sq, nb * 16, kk, lane, b);
                mma4(st[2 * nb], ka, b[0], b[1]);
                mma4(st[2 * nb + 1], ka, b[2], b[3]);
                ld_b(sg, nb * 16, kk, lane, b);
                mma4(dpt[2 * nb], va, b[0], b[1]);
                mma4(dpt[2 * nb + 1], va, b[2], b[3]);
            }
        }
        // P^T and dS^T: rows are keys k0 + g (+ 8), columns queries
        const bool kv0 = k0 + g < nkeys, kv1 = k0 + g + 8 < nkeys;
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int c = nt * 8 + 2 * tq + (e & 1);
                const bool ok = (e >> 1) ? kv1 : kv0;
                const float p = ok ? exp2f(st[nt][e] * sc2 - sL[c]) : 0.f;
                st[nt][e] = p;
                dpt[nt][e] = p * (dpt[nt][e] - sD[c]);
            }
        float dv[8][4], dk[8][4];
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
            for (int e = 0; e < 4; ++e) dv[i][e] = dk[i][e] = 0.f;
#pragma unroll
        for (int kq = 0; kq < NQ; ++kq) {
            uint32_t pa[4], da[4];
            acc_to_a(st[2 * kq], st[2 * kq + 1], pa);
            acc_to_a(dpt[2 * kq], dpt[2 * kq + 1], da);
#pragma unroll
            for (int dn = 0; dn < 4; ++dn) {
                uint32_t b[4];
                ld_bt(sg, kq * 16, dn, lane, b);
                mma4(dv[2 * dn], pa, b[0], b[1]);
                mma4(dv[2 * dn + 1], pa, b[2], b[3]);
                ld_bt(sq, kq * 16, dn, lane, b);
                mma4(dk[2 * dn], da, b[0], b[1]);
                mma4(dk[2 * dn + 1], da, b[2], b[3]);
            }
        }
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const int j = k0 + g + 8 * i;
            if (j >= nkeys) continue;
            uint16_t* kr = j < L ? dkvc + (size_t)(ctx0 + j) * 2 * dm + h * kHd
                                 : dqkv + (size_t)(act0 + j - L) * 3 * dm + dm + h * kHd;
#pragma unroll
            for (int nt = 0; nt < 8; ++nt) {
                *reinterpret_cast<uint32_t*>(kr + nt * 8 + 2 * tq) =
                    pack_bf2(dk[nt][2 * i] * sc, dk[nt][2 * i + 1] * sc);
                *reinterpret_cast<uint32_t*>(kr + dm + nt * 8 + 2 * tq) =
                    pack_bf2(dv[nt][2 * i], dv[nt][2 * i + 1]);
            }
        }
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
    // the row in registers: lane holds columns 8 lane + 256 i, i < dm / 256
    float xr[4][8];
#pragma unroll
    for (int i = 0; i < 4; ++i)
        if (256 * i < dm) {
            const uint4 q = *reinterpret_cast<const uint4*>(nf + (size_t)r * dm + 256 * i + 8 * lane);
            const uint32_t w4[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                xr[i][2 * e] = __uint_as_float(w4[e] << 16);
                xr[i][2 * e + 1] = __uint_as_float(w4[e] & 0xffff0000u);
            }
        }
    float sq = 0.f;
    for (int k = 0; k < D; ++k) {
        const uint16_t* wr = w_out + ((size_t)t * D + k) * dm + 8 * lane;
        float acc = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i)
            if (256 * i < dm) {
                const uint4 q = *reinterpret_cast<const uint4*>(wr + 256 * i);
                const uint32_t w4[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    acc = fmaf(xr[i][2 * e], __uint_as_float(w4[e] << 16), acc);
                    acc = fmaf(xr[i][2 * e + 1], __uint_as_float(w4[e] & 0xffff0000u), acc);
                }
            }
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

// dphi[s, j] = sum_c dh[s C + c, j] (the time embedding is added to every
// action row of the sample), c in order.
__global__ void __launch_bounds__(256) k_flow_dphi(const float* __restrict__ dh, FlowDims dd,
                                                   float* __restrict__ dphi) {
    const int s = blockIdx.x, dm = dd.dm, C = dd.C;
    const int j = blockIdx.y * blockDim.x + threadIdx.x;
    if (j >= dm) return;
    float acc = 0.f;
    for (int c = 0; c < C; ++c) acc += dh[((size_t)s * C + c) * dm + j];
    dphi[(size_t)s * dm + j] = acc;
}

// dz1[s, k] = (sum_j dphi[s, j] T2[j, k]) SiLU'(z1[s, k]) over (sample, block
// of 128 columns k).  Thread (jg, kq): 8 consecutive columns (one 16-byte load
// per row), rows j = jg, jg + 16, ...; the 16 row groups are summed in order.
__global__ void __launch_bounds__(256) k_flow_time_bwd(const int* __restrict__ sample_slot,
                                                       const __grid_constant__ FlowSlots fs,
                                                       FlowDims dd, const uint16_t* __restrict__ t2,
                                                       const float* __restrict__ z1,
                                                       const float* __restrict__ dphi,
                                                       float* __restrict__ dz1) {
    extern __shared__ float sh[];  // dphi [dm], then partials [16][128]
    const int s = blockIdx.x, dm = dd.dm, k0 = blockIdx.y * 128;
    const int t = fs.tenant[sample_slot[s]];
    for (int j = threadIdx.x; j < dm; j += blockDim.x) sh[j] = dphi[(size_t)s * dm + j];
    __syncthreads();
    const int jg = threadIdx.x >> 4, kq = threadIdx.x & 15;
    const uint16_t* T2 = t2 + (size_t)t * dm * dm + k0 + 8 * kq;
    float acc[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] = 0.f;
    for (int j = jg; j < dm; j += 16) {
        const uint4 q = *reinterpret_cast<const uint4*>(T2 + (size_t)j * dm);
        const uint32_t u[4] = {q.x, q.y, q.z, q.w};
        const float g = sh[j];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            acc[2 * e] = fmaf(g, __uint_as_float(u[e] << 16), acc[2 * e]);
            acc[2 * e + 1] = fmaf(g, __uint_as_float(u[e] & 0xffff0000u), acc[2 * e + 1]);
        }
    }
    float* part = sh + dm;
#pragma unroll
    for (int e = 0; e < 8; ++e) part[jg * 128 + 8 * kq + e] = acc[e];
    __syncthreads();
    if (threadIdx.x < 128) {
        float v = 0.f;
        for (int g = 0; g < 16; ++g) v += part[g * 128 + threadIdx.x];
        const size_t o = (size_t)s * dm + k0 + threadIdx.x;
        dz1[o] = v * silu_grad_f(z1[o]);
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
    // the context weight gradient on the tensor cores: the hidden rows and
    // dKV_c transposed, each tenant's rows at a 64-aligned column offset
    uint16_t *xT, *dkT;       // [d, kpad], [2 dm, kpad]
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

FlowWs carve_flow(const FlowDims& d, int S, int N, int n_slots, void* base) {
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
    const size_t kpad = (n + 63) / 64 * 64 + 64 * (size_t)std::max(n_slots, 0);
    w.xT = b16((size_t)d.d * kpad);
    w.dkT = b16(2 * dm * kpad);
    w.bytes = off;
    return w;
}

jnx_status last(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Query tiles of 16 rows: one tile -> four key slices per tile of 64 keys,
// two -> two, three or four -> one.
jnx_status flow_attn_fwd_launch(const uint16_t* qkv, const uint16_t* kvc, const int* cu,
                                const FlowDims& d, uint16_t* o, float* lse, int S,
                                cudaStream_t s) {
    if (S == 0) return JNX_OK;
    const int MT = (d.C + 15) / 16;
    const dim3 grid(S, d.nh);
    if (MT == 1)
        k_flow_attn_fwd<4><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, lse);
    else if (MT == 2)
        k_flow_attn_fwd<2><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, lse);
    else
        k_flow_attn_fwd<1><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, lse);
    return last("flow attention");
}

template <int NQ>
void launch_bwd_kv(dim3 grid, const uint16_t* qkv, const uint16_t* kvc, const int* cu,
                   const FlowDims& d, const uint16_t* o, const float* dO, const float* lse,
                   uint16_t* dqkv, uint16_t* dkvc, cudaStream_t s) {
    k_flow_attn_bwd_kv<NQ><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, dO, lse, dqkv, dkvc);
}

// dq (query side), then dk / dv (key side: one CTA per sample, head and
// key tile up to 16 tiles, striding beyond).
jnx_status flow_attn_bwd_launch(const uint16_t* qkv, const uint16_t* kvc, const jnx_group* g,
                                const FlowDims& d, const uint16_t* o, const float* dO,
                                const float* lse, uint16_t* dqkv, uint16_t* dkvc,
                                cudaStream_t s) {
    const int S = g->n_samples;
    if (S == 0) return JNX_OK;
    const int MT = (d.C + 15) / 16;
    const int* cu = g->cu_seqlens;
    const dim3 grid(S, d.nh);
    if (MT == 1)
        k_flow_attn_bwd_q<4><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, dO, lse, dqkv);
    else if (MT == 2)
        k_flow_attn_bwd_q<2><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, dO, lse, dqkv);
    else
        k_flow_attn_bwd_q<1><<<grid, 128, 0, s>>>(qkv, kvc, cu, d, o, dO, lse, dqkv);
    int tiles = 1;
    for (int i = 0; i < S; ++i)
        tiles = std::max(tiles, (g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i] + d.C + kKT - 1) / kKT);
    const dim3 gkv(S, d.nh, std::min(tiles, 16));
    switch (MT) {
        case 1: launch_bwd_kv<1>(gkv, qkv, kvc, cu, d, o, dO, lse, dqkv, dkvc, s); break;
        case 2: launch_bwd_kv<2>(gkv, qkv, kvc, cu, d, o, dO, lse, dqkv, dkvc, s); break;
        case 3: launch_bwd_kv<3>(gkv, qkv, kvc, cu, d, o, dO, lse, dqkv, dkvc, s); break;
        default: launch_bwd_kv<4>(gkv, qkv, kvc, cu, d, o, dO, lse, dqkv, dkvc, s); break;
    }
    return last("flow attention backward");
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
    if ((reinterpret_cast<uintptr_t>(fh->t1) | reinterpret_cast<uintptr_t>(fh->t2) |
         reinterpret_cast<uintptr_t>(fh->w_out)) & 15)
        return fail(JNX_ERR_INVALID_ARG, "flow: t1, t2 and w_out must be 16-byte aligned");
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
            if ((st = flow_attn_fwd_launch(qkv, kvc, g->cu_seqlens, d, o, lse, S, s))) return st;
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
    return carve_flow(d, g->n_samples, g->n_tokens, g->n_slots, nullptr).bytes;
}

static jnx_status flow_begin(const jnx_flow_head* fh, const jnx_group* g, const uint16_t* hidden,
                             void* workspace, size_t ws_bytes, FlowDims& d, FlowWs& w) {
    jnx_status st;
    if ((st = check_flow(fh, g, d))) return st;
    if (!workspace || (g->n_tokens > 0 && !hidden))
        return fail(JNX_ERR_INVALID_ARG, "flow: null workspace or hidden rows");
    if (reinterpret_cast<uintptr_t>(workspace) & 255)
        return fail(JNX_ERR_INVALID_ARG, "flow: workspace must be 256-byte aligned");
    w = carve_flow(d, g->n_samples, g->n_tokens, g->n_slots, workspace);
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
    const dim3 tg(S, d.dm / kTimeRows);
    k_flow_time1<<<tg, 256, d.dm * sizeof(float), s>>>(tau, g->sample_slot, fs, d, fh->t1, fh->tb1,
                                                       w.sfeat, w.z1);
    k_flow_time2<<<tg, 256, d.dm * sizeof(float), s>>>(g->sample_slot, fs, d, fh->t2, fh->tb2,
                                                       w.z1, w.phi);
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
    // the context weight gradient dW_kvc[t] = dKV_c^T X over tenant t's token
    // rows runs as one tcgen05 GEMM per tenant (K = its rows, padded to 64)
    // on transposed copies; widths that are not a multiple of 256 keep the
    // mma.sync segmented kernel
    const bool tc_kvc = d.d % 256 == 0;
    static thread_local SegRows rp;  // token-row segments at padded offsets
    rp = rt;
    std::vector<int> kp(nsl);
    int kpad = 0;
    for (int i = 0; i < nsl; ++i) {
        rp.tile_start[i] = kpad;
        kp[i] = (rt.r1[i] - rt.r0[i] + 63) / 64 * 64;
        kpad += kp[i];
    }
    if (tc_kvc && (st = transpose_seg_launch(hidden, d.d, d.d, rp, kpad, w.xT, s))) return st;
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
            if ((st = flow_attn_bwd_launch(qkv, kvc, g, d, o, w.dO, lse, w.dqkv, w.dkvc, s)))
                return st;
        }
        {
            TraceScope ts(JNX_K_FLOW_WGRAD,
                          2.0 * Ma * 3 * dm * dm + 2.0 * g->n_tokens * 2 * dm * d.d, s);
            if ((st = seg_wgrad_launch(ra, w.dqkv, 3 * dm, n1, dm, 3 * dm, dm, G.w_qkv,
                                       (long long)3 * dm * dm, add, s)))
                return st;
            if (!tc_kvc) {
                if ((st = seg_wgrad_launch(rt, w.dkvc, 2 * dm, hidden, d.d, 2 * dm, d.d,
                                           G.w_kvc, (long long)2 * dm * d.d, add, s)))
                    return st;
            } else {
                if ((st = transpose_seg_launch(w.dkvc, 2 * dm, 2 * dm, rp, kpad, w.dkT, s)))
                    return st;
                for (int i = 0; i < nsl; ++i) {
                    float* gw = G.w_kvc + (size_t)rt.tenant[i] * 2 * dm * d.d;
                    if (kp[i] == 0) {  // no context rows: a zero gradient
                        if (!add && cudaMemsetAsync(gw, 0, sizeof(float) * 2 * dm * d.d, s))
                            return last("flow context weight gradient");
                        continue;
                    }
                    GemmParams q{};
                    q.M = 2 * dm;
                    q.N = d.d;
                    q.K = kp[i];
                    q.status = w.status;
                    if (add) {
                        q.epi = EPI_RESID;
                        q.resid = gw;
                        q.ldr = d.d;
                    } else {
                        q.epi = EPI_F32;
                        q.out = gw;
                        q.ldo = d.d;
                    }
                    if ((st = gemm_launch(w.dkT + rp.tile_start[i], kpad, w.xT + rp.tile_start[i],
                                          kpad, q, s)))
                        return st;
                }
            }
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
    k_flow_dphi<<<dim3(S, (dm + 255) / 256), 256, 0, s>>>(w.dh, d, w.dphi);
    k_flow_time_bwd<<<dim3(S, dm / 128), 256, (dm + 16 * 128) * sizeof(float), s>>>(
        g->sample_slot, fs, d, fh->t2, w.z1, w.dphi, w.dz1);
    k_flow_outer<true><<<dim3(nsl, dm), 256, 0, s>>>(w.dphi, w.z1, fs, d, gr->t2, gr->tb2, add);
    k_flow_outer<false><<<dim3(nsl, dm), 256, 0, s>>>(w.dz1, w.sfeat, fs, d, gr->t1, gr->tb1, add);
    return last("flow embedding backward");
}
