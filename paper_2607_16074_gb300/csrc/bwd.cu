// Kernels of the per-tenant LoRA backward through the frozen backbone that
// are not GEMM- or attention-shaped:
//
//   k_transpose     bf16 [batch][rows][cols] -> [batch][cols][rows] (the
//                   frozen weights' transposes, read by the input-gradient
//                   GEMMs; the adapters' B^T each step)
//   k_rms_bwd       RMSNorm backward with the residual gradient added (one
//                   warp per row; k_rms_bwd_row, one CTA per row with the
//                   row in registers, for 1024 <= d <= 4096)
//   k_attn_bwd_prep attention's dO in bf16 and D = rowsum(dO * O) per head
//   k_seg_up        per tenant segment  out[rows] (+)= sum_p T_p W_p[t]
//                   (LoRA up-projections of gradients; the query heads'
//                   feature gradient), bf16 mma.sync
//   k_seg_tn        per row chunk  U^T V  (LoRA weight gradients reduce over
//                   a tenant's rows), bf16 mma.sync, then k_seg_reduce adds
//                   a tenant's chunks in a fixed order
//   k_mlp_dfeat     MLP heads: dloss/d(final normed row) = (dz W1) / L
//
// The rank-16 products are skinny (one side 16 wide), so they run on the
// warp-level mma.sync path; the dense input-gradient GEMMs are tcgen05
// (gemm.cu) and attention's backward is tcgen05 (attn_bwd.cu).
#include <algorithm>
#include <vector>

#include "jnx_bwd.h"
#include "jnx_dev.cuh"

namespace jnx {

// ---------------------------------------------------------------------------
// transpose
// ---------------------------------------------------------------------------
// 64 x 64 tiles through shared memory, 16-byte loads along the source rows
// and 16-byte stores along the destination rows when the buffers are 16-byte
// aligned (vec), element by element at the edges and otherwise.
__global__ void __launch_bounds__(256) k_transpose(const uint16_t* __restrict__ src, int rows,
                                                   int cols, uint16_t* __restrict__ dst, int vec) {
    __shared__ uint16_t tile[64][64 + 2];
    const size_t plane = (size_t)rows * cols;
    src += (size_t)blockIdx.z * plane;
    dst += (size_t)blockIdx.z * plane;
    const int r0 = blockIdx.y * 64, c0 = blockIdx.x * 64;
    const bool vec_in = vec && (cols % 8) == 0 && c0 + 64 <= cols;
    for (int i = threadIdx.x; i < 64 * 8; i += 256) {
        const int r = i / 8, u = i % 8;  // 8 elements at columns c0 + 8 u
        if (r0 + r >= rows) continue;
        if (vec_in) {
            const uint4 v = *reinterpret_cast<const uint4*>(src + (size_t)(r0 + r) * cols + c0 + 8 * u);
            const uint16_t* e = reinterpret_cast<const uint16_t*>(&v);
#pragma unroll
            for (int k = 0; k < 8; ++k) tile[r][8 * u + k] = e[k];
        } else {
            for (int k = 0; k < 8; ++k) {
                const int c = c0 + 8 * u + k;
                if (c < cols) tile[r][8 * u + k] = src[(size_t)(r0 + r) * cols + c];
            }
        }
    }
    __syncthreads();
    const bool vec_out = vec && (rows % 8) == 0 && r0 + 64 <= rows;
    for (int i = threadIdx.x; i < 64 * 8; i += 256) {
        const int c = i / 8, u = i % 8;  // destination row c0 + c, columns r0 + 8 u
        if (c0 + c >= cols) continue;
        if (vec_out) {
            uint16_t e[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) e[k] = tile[8 * u + k][c];
            *reinterpret_cast<uint4*>(dst + (size_t)(c0 + c) * rows + r0 + 8 * u) =
                *reinterpret_cast<const uint4*>(e);
        } else {
            for (int k = 0; k < 8; ++k) {
                const int r = r0 + 8 * u + k;
                if (r < rows) dst[(size_t)(c0 + c) * rows + r] = tile[8 * u + k][c];
            }
        }
    }
}

jnx_status transpose_launch(const uint16_t* src, int batch, int rows, int cols, uint16_t* dst,
                            cudaStream_t s) {
    if (batch < 0 || rows < 0 || cols < 0) return fail(JNX_ERR_INVALID_ARG, "transpose: sizes");
    if (batch == 0 || rows == 0 || cols == 0) return JNX_OK;
    if ((rows + 63) / 64 > 65535 || batch > 65535)
        return fail(JNX_ERR_UNSUPPORTED, "transpose: too many rows or planes");
    const int vec = ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0;
    k_transpose<<<dim3((cols + 63) / 64, (rows + 63) / 64, batch), 256, 0, s>>>(src, rows, cols,
                                                                             dst, vec);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "transpose: %s", cudaGetErrorString(e));
}

// Segment-padded transpose: dst [cols][kpad] bf16 with dst[c][p] = src[r][c]
// for the row r that padded position p stands for: segment i's rows
// r0_i .. r1_i - 1 sit at positions off_i .. off_i + (r1_i - r0_i) - 1
// (off_i = sr.tile_start[i], ascending, 64-aligned), every other position is
// zero.  64 x 64 tiles as k_transpose (cols % 64 == 0, kpad % 64 == 0,
// 16-byte aligned buffers and strides).
__global__ void __launch_bounds__(256) k_transpose_seg(const uint16_t* __restrict__ src, int ld_src,
                                                       const __grid_constant__ SegRows sr, int kpad,
                                                       uint16_t* __restrict__ dst) {
    __shared__ uint16_t tile[64][64 + 2];
    __shared__ int srow[64];
    const int p0 = blockIdx.y * 64, c0 = blockIdx.x * 64;
    if (threadIdx.x < 64) {
        const int p = p0 + threadIdx.x;
        int lo = 0, hi = sr.n - 1;  // last segment with off <= p
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (sr.tile_start[mid] <= p) lo = mid; else hi = mid - 1;
        }
        const int r = sr.r0[lo] + (p - sr.tile_start[lo]);
        srow[threadIdx.x] = (sr.n > 0 && p >= sr.tile_start[lo] && r < sr.r1[lo]) ? r : -1;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 64 * 8; i += 256) {
        const int rr = i / 8, u = i % 8;
        const int r = srow[rr];
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (r >= 0) v = *reinterpret_cast<const uint4*>(src + (size_t)r * ld_src + c0 + 8 * u);
        const uint16_t* e = reinterpret_cast<const uint16_t*>(&v);
#pragma unroll
        for (int k = 0; k < 8; ++k) tile[rr][8 * u + k] = e[k];
    }
    __syncthreads();
    for (int i = threadIdx.x; i < 64 * 8; i += 256) {
        const int c = i / 8, u = i % 8;
        uint16_t e[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) e[k] = tile[8 * u + k][c];
        *reinterpret_cast<uint4*>(dst + (size_t)(c0 + c) * kpad + p0 + 8 * u) =
            *reinterpret_cast<const uint4*>(e);
    }
}

jnx_status transpose_seg_launch(const uint16_t* src, int ld_src, int cols, const SegRows& sr,
                                int kpad, uint16_t* dst, cudaStream_t s) {
    if (cols <= 0 || cols % 64 || kpad % 64 || ld_src % 8 ||
        ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15))
        return fail(JNX_ERR_UNSUPPORTED, "segmented transpose: layout");
    if (kpad == 0) return JNX_OK;
    if (kpad / 64 > 65535) return fail(JNX_ERR_UNSUPPORTED, "segmented transpose: too many rows");
    k_transpose_seg<<<dim3(cols / 64, kpad / 64), 256, 0, s>>>(src, ld_src, sr, kpad, dst);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "segmented transpose: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// RMSNorm backward: with s = rsqrt(mean(x^2) + eps) and n = x s gamma,
//   dx = dres + s (gamma dn) - x s^3 mean(gamma dn x)
// One warp per row; dres (may be null, may alias dx) is the gradient that
// reaches x along the residual path.  Also writes bf16(dx) when dx_bf is set.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_rms_bwd(const float* __restrict__ x,
                                                 const uint16_t* __restrict__ gamma, float eps,
                                                 const float* __restrict__ dn, const float* dres,
                                                 int M, int d, float* dx, uint16_t* dx_bf) {
    const int row = blockIdx.x * 8 + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    if (row >= M) return;
    const float* xr = x + (size_t)row * d;
    const float* dr = dn + (size_t)row * d;
    float ss = 0.f, sd = 0.f;
    for (int c = lane * 4; c < d; c += 128) {
        const float4 xv = *reinterpret_cast<const float4*>(xr + c);
        const float4 dv = *reinterpret_cast<const float4*>(dr + c);
        const uint2 g = *reinterpret_cast<const uint2*>(gamma + c);
        ss += xv.x * xv.x + xv.y * xv.y + xv.z * xv.z + xv.w * xv.w;
        sd += bf2f(g.x & 0xFFFF) * dv.x * xv.x + bf2f(g.x >> 16) * dv.y * xv.y +
              bf2f(g.y & 0xFFFF) * dv.z * xv.z + bf2f(g.y >> 16) * dv.w * xv.w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        ss += __shfl_xor_sync(0xffffffffu, ss, o);
        sd += __shfl_xor_sync(0xffffffffu, sd, o);
    }
    const float s = rsqrtf(ss / (float)d + eps);
    const float k = s * s * s * sd / (float)d;
    for (int c = lane * 4; c < d; c += 128) {
        const float4 xv = *reinterpret_cast<const float4*>(xr + c);
        const float4 dv = *reinterpret_cast<const float4*>(dr + c);
        const uint2 g = *reinterpret_cast<const uint2*>(gamma + c);
        float4 r = dres ? *reinterpret_cast<const float4*>(dres + (size_t)row * d + c)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        r.x += s * bf2f(g.x & 0xFFFF) * dv.x - xv.x * k;
        r.y += s * bf2f(g.x >> 16) * dv.y - xv.y * k;
        r.z += s * bf2f(g.y & 0xFFFF) * dv.z - xv.z * k;
        r.w += s * bf2f(g.y >> 16) * dv.w - xv.w * k;
        *reinterpret_cast<float4*>(dx + (size_t)row * d + c) = r;
        if (dx_bf)
            *reinterpret_cast<uint2*>(dx_bf + (size_t)row * d + c) =
                make_uint2(pack_bf2(r.x, r.y), pack_bf2(r.z, r.w));
    }
}

// The same for 1024 <= d <= 4096: one 256-thread CTA per row, each thread
// holding NU float4 units of x and dn (units tid, tid + 256, ...) in
// registers, so every input byte is read once; the row sums are combined
// over the warps in a fixed order.
template <int NU>
__global__ void __launch_bounds__(256) k_rms_bwd_row(const float* __restrict__ x,
                                                     const uint16_t* __restrict__ gamma, float eps,
                                                     const float* __restrict__ dn, const float* dres,
                                                     int d, float* dx, uint16_t* dx_bf) {
    __shared__ float red[2][8];
    const size_t row = blockIdx.x;
    const int units = d / 4, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const float* xr = x + row * d;
    const float* dr = dn + row * d;
    float4 xv[NU], dv[NU];
    uint2 gv[NU];
    float ss = 0.f, sd = 0.f;
#pragma unroll
    for (int i = 0; i < NU; ++i) {
        const int u = threadIdx.x + 256 * i;
        xv[i] = dv[i] = make_float4(0.f, 0.f, 0.f, 0.f);
        gv[i] = make_uint2(0u, 0u);
        if (u < units) {
            xv[i] = *reinterpret_cast<const float4*>(xr + 4 * u);
            dv[i] = *reinterpret_cast<const float4*>(dr + 4 * u);
            gv[i] = *reinterpret_cast<const uint2*>(gamma + 4 * u);
        }
        ss += xv[i].x * xv[i].x + xv[i].y * xv[i].y + xv[i].z * xv[i].z + xv[i].w * xv[i].w;
        sd += bf2f(gv[i].x & 0xFFFF) * dv[i].x * xv[i].x + bf2f(gv[i].x >> 16) * dv[i].y * xv[i].y +
              bf2f(gv[i].y & 0xFFFF) * dv[i].z * xv[i].z + bf2f(gv[i].y >> 16) * dv[i].w * xv[i].w;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        ss += __shfl_xor_sync(0xffffffffu, ss, o);
        sd += __shfl_xor_sync(0xffffffffu, sd, o);
    }
    if (lane == 0) {
        red[0][warp] = ss;
        red[1][warp] = sd;
    }
    __syncthreads();
    ss = sd = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) {
        ss += red[0][w];
        sd += red[1][w];
    }
    const float s = rsqrtf(ss / (float)d + eps);
    const float k = s * s * s * sd / (float)d;
#pragma unroll
    for (int i = 0; i < NU; ++i) {
        const int u = threadIdx.x + 256 * i;
        if (u >= units) continue;
        float4 r = dres ? *reinterpret_cast<const float4*>(dres + row * d + 4 * u)
                        : make_float4(0.f, 0.f, 0.f, 0.f);
        r.x += s * bf2f(gv[i].x & 0xFFFF) * dv[i].x - xv[i].x * k;
        r.y += s * bf2f(gv[i].x >> 16) * dv[i].y - xv[i].y * k;
        r.z += s * bf2f(gv[i].y & 0xFFFF) * dv[i].z - xv[i].z * k;
        r.w += s * bf2f(gv[i].y >> 16) * dv[i].w - xv[i].w * k;
        *reinterpret_cast<float4*>(dx + row * d + 4 * u) = r;
        if (dx_bf)
            *reinterpret_cast<uint2*>(dx_bf + row * d + 4 * u) =
                make_uint2(pack_bf2(r.x, r.y), pack_bf2(r.z, r.w));
    }
}

jnx_status rms_bwd_launch(const float* x, const uint16_t* gamma, float eps, const float* dn,
                          const float* dres, int M, int d, float* dx, uint16_t* dx_bf,
                          cudaStream_t s) {
    if (d % 128) return fail(JNX_ERR_UNSUPPORTED, "rms backward: d %% 128 != 0");
    if (M <= 0) return JNX_OK;
    if (d >= 1024 && d <= 4096) {
        if (d <= 1024)
            k_rms_bwd_row<1><<<M, 256, 0, s>>>(x, gamma, eps, dn, dres, d, dx, dx_bf);
        else if (d <= 2048)
            k_rms_bwd_row<2><<<M, 256, 0, s>>>(x, gamma, eps, dn, dres, d, dx, dx_bf);
        else
            k_rms_bwd_row<4><<<M, 256, 0, s>>>(x, gamma, eps, dn, dres, d, dx, dx_bf);
    } else {
        k_rms_bwd<<<(M + 7) / 8, 256, 0, s>>>(x, gamma, eps, dn, dres, M, d, dx, dx_bf);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "rms backward: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// Attention backward prologue: dO = bf16(datt), D[row, h] = sum over head h's
// columns of dO * O (both as the bf16 values the backward kernels read).
// One warp per (row, head).
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_attn_bwd_prep(const float* __restrict__ datt,
                                                       const uint16_t* __restrict__ att, int M,
                                                       int H, int hd, uint16_t* __restrict__ dO,
                                                       float* __restrict__ D) {
    const long long w = (long long)blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (w >= (long long)M * H) return;
    const int row = (int)(w / H), h = (int)(w % H);
    const size_t base = (size_t)row * H * hd + (size_t)h * hd;
    float acc = 0.f;
    for (int c = lane * 4; c < hd; c += 128) {
        const float4 g = *reinterpret_cast<const float4*>(datt + base + c);
        const uint2 o = *reinterpret_cast<const uint2*>(att + base + c);
        const uint32_t p0 = pack_bf2(g.x, g.y), p1 = pack_bf2(g.z, g.w);
        *reinterpret_cast<uint2*>(dO + base + c) = make_uint2(p0, p1);
        acc += bf2f(p0 & 0xFFFF) * bf2f(o.x & 0xFFFF) + bf2f(p0 >> 16) * bf2f(o.x >> 16) +
               bf2f(p1 & 0xFFFF) * bf2f(o.y & 0xFFFF) + bf2f(p1 >> 16) * bf2f(o.y >> 16);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) D[(size_t)row * H + h] = acc;
}

jnx_status attn_bwd_prep_launch(const float* datt, const uint16_t* att, int M, int H, int hd,
                                uint16_t* dO, float* D, cudaStream_t s) {
    if (hd % 128 && hd != 64) return fail(JNX_ERR_UNSUPPORTED, "attention prep: head dim");
    if (M <= 0) return JNX_OK;
    const long long warps = (long long)M * H;
    k_attn_bwd_prep<<<(unsigned)((warps + 7) / 8), 256, 0, s>>>(datt, att, M, H, hd, dO, D);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "attention prep: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// Segmented products on mma.sync (m16n8k16, bf16 in, fp32 accumulate).
// Shared-memory tiles are stored in 16-byte units XOR-swizzled by row so
// ldmatrix reads of 8 rows hit distinct banks.
// ---------------------------------------------------------------------------
namespace seg {
constexpr int UP_BM = 64, UP_BN = 128, UP_BK = 16;
constexpr int TN_ROWS = 32, TN_BN = 256;
}  // namespace seg

// out[row, c] (+)= sum_p sum_k T_p[row, k] W_p[tenant(row)][k, c]: CTA tile
// 64 rows x 128 columns, 4 warps as 2 x 2 (32 x 64 each), k in steps of 16
// across the parts.  W_p[t] is row-major [k_p, ncols] at w + t * wstride.
// T_p tile: 64 rows x 32 bytes; W tile: 16 k-rows x 256 bytes.
template <bool ADD>
__global__ void __launch_bounds__(128) k_seg_up(const __grid_constant__ SegRows sr,
                                                const __grid_constant__ SegUpParts sp, int ncols,
                                                float* __restrict__ out, int ldo) {
    using namespace seg;
    __shared__ __align__(128) uint8_t sT[2][UP_BM * 32];
    __shared__ __align__(128) uint8_t sW[2][UP_BK * 256];
    int sg = 0;
    while (sg + 1 < sr.n && sr.tile_start[sg + 1] <= (int)blockIdx.x) ++sg;
    const int r1 = sr.r1[sg];
    const int row0 = sr.r0[sg] + ((int)blockIdx.x - sr.tile_start[sg]) * UP_BM;
    if (row0 >= r1) return;
    if (sp.w[0][sg] == nullptr) return;  // not this launch's slot
    const int c0 = blockIdx.y * UP_BN;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wm = warp & 1, wn = warp >> 1;
    const uint32_t ta = smem_u32(sT), wa = smem_u32(sW);
    int nsteps = 0;
    for (int p = 0; p < sp.n_parts; ++p) nsteps += sp.k[p] / UP_BK;
    auto step_part = [&](int st, int& p, int& k0) {
        p = 0;
        k0 = st * UP_BK;
        while (k0 >= sp.k[p]) {
            k0 -= sp.k[p];
            ++p;
        }
    };
    auto load = [&](int st, int buf) {
        int p, k0;
        step_part(st, p, k0);
        {   // T: 64 rows x 2 units
            const int r = tid >> 1, u = tid & 1;
            const bool ok = row0 + r < r1;
            const uint16_t* src = sp.t[p] + (size_t)(ok ? row0 + r : row0) * sp.ldt[p] + k0 + u * 8;
            cp_async16(ta + buf * UP_BM * 32 + r * 32 + ((u ^ ((r >> 2) & 1)) << 4), src, ok);
        }
        const uint16_t* wsrc = sp.w[p][sg];
        for (int i = tid; i < UP_BK * 16; i += 128) {  // W: 16 rows x 16 units
            const int r = i >> 4, u = i & 15;
            cp_async16(wa + buf * UP_BK * 256 + r * 256 + ((u ^ (r & 7)) << 4),
                       wsrc + (size_t)(k0 + r) * ncols + c0 + u * 8, true);
        }
    };
    float acc[2][8][4];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j][0] = acc[i][j][1] = acc[i][j][2] = acc[i][j][3] = 0.f;
    const int mi = lane >> 3, rr = lane & 7;
    load(0, 0);
    cp_async_commit();
    for (int st = 0; st < nsteps; ++st) {
        const int buf = st & 1;
        if (st + 1 < nsteps) load(st + 1, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t tb = ta + buf * UP_BM * 32, wb = wa + buf * UP_BK * 256;
        uint32_t a[2][4];
#pragma unroll
        for (int m = 0; m < 2; ++m) {
            const int r = wm * 32 + m * 16 + rr + 8 * (mi & 1), u = mi >> 1;
            ldsm_x4(tb + r * 32 + ((u ^ ((r >> 2) & 1)) << 4), a[m][0], a[m][1], a[m][2], a[m][3]);
        }
#pragma unroll
        for (int nb = 0; nb < 4; ++nb) {
            const int r = rr + 8 * (mi & 1), u = wn * 8 + nb * 2 + (mi >> 1);
            uint32_t b0, b1, b2, b3;
            ldsm_x4_t(wb + r * 256 + ((u ^ (r & 7)) << 4), b0, b1, b2, b3);
#pragma unroll
            for (int m = 0; m < 2; ++m) {
                mma_bf16(acc[m][2 * nb], a[m][0], a[m][1], a[m][2], a[m][3], b0, b1);
                mma_bf16(acc[m][2 * nb + 1], a[m][0], a[m][1], a[m][2], a[m][3], b2, b3);
            }
        }
        __syncthreads();
    }
    const int g = lane >> 2, q = lane & 3;
#pragma unroll
    for (int m = 0; m < 2; ++m)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int row = row0 + wm * 32 + m * 16 + g + 8 * h;
            if (row >= r1) continue;
            float* o = out + (size_t)row * ldo + c0 + wn * 64 + 2 * q;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                float2 v = make_float2(acc[m][j][2 * h], acc[m][j][2 * h + 1]);
                if (ADD) {
                    const float2 old = *reinterpret_cast<const float2*>(o + j * 8);
                    v.x += old.x;
                    v.y += old.y;
                }
                *reinterpret_cast<float2*>(o + j * 8) = v;
            }
        }
}

// Partial sums over one row chunk [cr0, cr1) of one tenant:
//   part[chunk][j][c] = sum_rows U[row, j] V[row, c],  j < 16, c in the
// CTA's 256 columns.  4 warps x 64 columns; rows in steps of 32 (two k16
// steps), double-buffered.
__global__ void __launch_bounds__(128) k_seg_tn(const __grid_constant__ SegChunks ch,
                                                const uint16_t* __restrict__ U, int ldu,
                                                const uint16_t* __restrict__ V, int ldv, int n,
                                                float* __restrict__ part) {
    using namespace seg;
    __shared__ __align__(128) uint8_t sU[2][TN_ROWS * 32];
    __shared__ __align__(128) uint8_t sV[2][TN_ROWS * 512];
    const int chunk = blockIdx.x;
    const int cr0 = ch.r0[chunk], cr1 = ch.r1[chunk];
    const int c0 = blockIdx.y * TN_BN;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t ua = smem_u32(sU), va = smem_u32(sV);
    const int nsteps = (cr1 - cr0 + TN_ROWS - 1) / TN_ROWS;
    auto load = [&](int st, int buf) {
        const int rbase = cr0 + st * TN_ROWS;
        if (tid < 64) {  // U: 32 rows x 2 units
            const int r = tid >> 1, u = tid & 1;
            const bool ok = rbase + r < cr1;
            cp_async16(ua + buf * TN_ROWS * 32 + r * 32 + ((u ^ ((r >> 2) & 1)) << 4),
                       U + (size_t)(ok ? rbase + r : cr0) * ldu + u * 8, ok);
        }
        for (int i = tid; i < TN_ROWS * 32; i += 128) {  // V: 32 rows x 32 units
            const int r = i >> 5, u = i & 31;
            const bool ok = rbase + r < cr1;
            cp_async16(va + buf * TN_ROWS * 512 + r * 512 + ((u ^ (r & 7)) << 4),
                       V + (size_t)(ok ? rbase + r : cr0) * ldv + c0 + u * 8, ok);
        }
    };
    float acc[8][4];
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
    const int mi = lane >> 3, rr = lane & 7;
    if (nsteps > 0) load(0, 0);
    cp_async_commit();
    for (int st = 0; st < nsteps; ++st) {
        const int buf = st & 1;
        if (st + 1 < nsteps) load(st + 1, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t ub = ua + buf * TN_ROWS * 32, vb = va + buf * TN_ROWS * 512;
#pragma unroll
        for (int ks = 0; ks < 2; ++ks) {
            // A = U^T (16 x 16 rows): transposed 8x8 blocks of U
            uint32_t a0, a1, a2, a3;
            {
                const int r = ks * 16 + rr + 8 * (mi >> 1), u = mi & 1;
                ldsm_x4_t(ub + r * 32 + ((u ^ ((r >> 2) & 1)) << 4), a0, a1, a2, a3);
            }
#pragma unroll
            for (int nb = 0; nb < 4; ++nb) {
                const int r = ks * 16 + rr + 8 * (mi & 1), u = warp * 8 + nb * 2 + (mi >> 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vb + r * 512 + ((u ^ (r & 7)) << 4), b0, b1, b2, b3);
                mma_bf16(acc[2 * nb], a0, a1, a2, a3, b0, b1);
                mma_bf16(acc[2 * nb + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        __syncthreads();
    }
    const int g = lane >> 2, q = lane & 3;
    float* o = part + (size_t)chunk * 16 * n + c0 + warp * 64 + 2 * q;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        *reinterpret_cast<float2*>(o + (size_t)g * n + j * 8) = make_float2(acc[j][0], acc[j][1]);
        *reinterpret_cast<float2*>(o + (size_t)(g + 8) * n + j * 8) =
            make_float2(acc[j][2], acc[j][3]);
    }
}

// G[t] = sum of the tenant's chunk partials in chunk order, written (or
// added) to the tenant's gradient slice: [16, n] (TRANS = false) or [n, 16].
template <bool TRANS>
__global__ void __launch_bounds__(256) k_seg_reduce(const __grid_constant__ SegChunks ch,
                                                    const float* __restrict__ part, int n,
                                                    float* __restrict__ grad, long long gstride,
                                                    int add) {
    const int slot = blockIdx.y;
    const long long e = (long long)blockIdx.x * 256 + threadIdx.x;
    if (e >= 16LL * n) return;
    const int j = (int)(e / n), c = (int)(e % n);
    float s = 0.f;
    for (int k = ch.slot_chunk0[slot]; k < ch.slot_chunk0[slot + 1]; ++k)
        s += part[(size_t)k * 16 * n + (size_t)j * n + c];
    float* gp = grad + (size_t)ch.slot_tenant[slot] * gstride +
                (TRANS ? (size_t)c * 16 + j : (size_t)j * n + c);
    *gp = add ? *gp + s : s;
}

jnx_status seg_rows_build(const jnx_group* g, int bm, SegRows& sr, int& tiles) {
    if (g->n_slots > kSegMaxSlots) return fail(JNX_ERR_UNSUPPORTED, "segments: too many tenants");
    sr = SegRows{};
    sr.n = g->n_slots;
    tiles = 0;
    for (int i = 0; i < g->n_slots; ++i) {
        sr.tenant[i] = g->h_slot_tenant[i];
        sr.r0[i] = g->h_cu_seqlens[g->h_seg_offsets[i]];
        sr.r1[i] = g->h_cu_seqlens[g->h_seg_offsets[i + 1]];
        sr.tile_start[i] = tiles;
        tiles += (sr.r1[i] - sr.r0[i] + bm - 1) / bm;
    }
    return JNX_OK;
}

void seg_up_weights(const jnx_group* g, SegUpParts& sp, int part, const uint16_t* base,
                    long long stride) {
    for (int i = 0; i < g->n_slots && i < kSegMaxSlots; ++i)
        sp.w[part][i] = base + (size_t)g->h_slot_tenant[i] * stride;
}

jnx_status seg_up_launch(const jnx_group* g, const SegUpParts& sp, int ncols, float* out, int ldo,
                         bool add, cudaStream_t s) {
    if (ncols % seg::UP_BN || ldo % 2)
        return fail(JNX_ERR_UNSUPPORTED, "segmented up-projection: %d columns", ncols);
    for (int p = 0; p < sp.n_parts; ++p)
        if (sp.k[p] <= 0 || sp.k[p] % seg::UP_BK || sp.ldt[p] % 8)
            return fail(JNX_ERR_UNSUPPORTED, "segmented up-projection: part %d", p);
    SegRows sr;
    int tiles;
    jnx_status st = seg_rows_build(g, seg::UP_BM, sr, tiles);
    if (st) return st;
    if (tiles == 0) return JNX_OK;
    const dim3 grid(tiles, ncols / seg::UP_BN);
    if (add)
        k_seg_up<true><<<grid, 128, 0, s>>>(sr, sp, ncols, out, ldo);
    else
        k_seg_up<false><<<grid, 128, 0, s>>>(sr, sp, ncols, out, ldo);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "segmented up-projection: %s", cudaGetErrorString(e));
}

size_t seg_tn_part_floats(int n_tokens, int n_slots, int n) {
    const int chunk = std::max(kSegChunkRows, (n_tokens + kSegMaxChunks / 2 - 1) / (kSegMaxChunks / 2));
    const size_t chunks = (size_t)n_tokens / chunk + (size_t)n_slots + 1;
    return chunks * 16 * (size_t)n;
}

jnx_status seg_tn_launch(const jnx_group* g, const uint16_t* U, int ldu, const uint16_t* V,
                         int ldv, int n, float* part, size_t part_floats, float* grad,
                         long long gstride, bool trans, bool add, cudaStream_t s) {
    if (n % seg::TN_BN || ldu % 8 || ldv % 8)
        return fail(JNX_ERR_UNSUPPORTED, "adapter gradient: %d columns", n);
    if (g->n_slots > kSegMaxSlots) return fail(JNX_ERR_UNSUPPORTED, "segments: too many tenants");
    // row chunks of each tenant segment, long enough that the chunk count
    // stays within kSegMaxChunks
    const int chunk = std::max(kSegChunkRows,
                               (g->n_tokens + kSegMaxChunks / 2 - 1) / (kSegMaxChunks / 2));
    static thread_local SegChunks ch;
    ch = SegChunks{};
    ch.n_slots = g->n_slots;
    int nc = 0;
    for (int i = 0; i < g->n_slots; ++i) {
        ch.slot_tenant[i] = g->h_slot_tenant[i];
        ch.slot_chunk0[i] = nc;
        const int r0 = g->h_cu_seqlens[g->h_seg_offsets[i]];
        const int r1 = g->h_cu_seqlens[g->h_seg_offsets[i + 1]];
        for (int r = r0; r < r1; r += chunk) {
            if (nc >= kSegMaxChunks) return fail(JNX_ERR_UNSUPPORTED, "adapter gradient: chunks");
            ch.r0[nc] = r;
            ch.r1[nc] = std::min(r + chunk, r1);
            ++nc;
        }
    }
    ch.slot_chunk0[g->n_slots] = nc;
    if ((size_t)nc * 16 * n > part_floats)
        return fail(JNX_ERR_WORKSPACE, "adapter gradient: partial buffer too small");
    if (nc > 0) k_seg_tn<<<dim3(nc, n / seg::TN_BN), 128, 0, s>>>(ch, U, ldu, V, ldv, n, part);
    if (g->n_slots > 0) {
        const dim3 grid((unsigned)((16LL * n + 255) / 256), g->n_slots);
        if (trans)
            k_seg_reduce<true><<<grid, 256, 0, s>>>(ch, part, n, grad, gstride, add ? 1 : 0);
        else
            k_seg_reduce<false><<<grid, 256, 0, s>>>(ch, part, n, grad, gstride, add ? 1 : 0);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "adapter gradient: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// Weight gradient of a per-tenant linear layer: for every group tenant t,
//   G[t][m, n] (+)= sum over the tenant's rows of U[row, m] V[row, n]
// (U = the output gradient, V = the layer's input, both bf16).  One CTA per
// (segment, 64 x 128 tile of G) walks all of the segment's rows in order
// (no split over rows, so no partial sums and a fixed order); 4 warps as
// 2 (m) x 2 (n), 32 x 64 each; rows in steps of 32, double-buffered.
// ---------------------------------------------------------------------------
namespace seg {
constexpr int WG_BM = 64, WG_BN = 128, WG_ROWS = 32;
}

__global__ void __launch_bounds__(128) k_seg_wgrad(const __grid_constant__ SegRows sr,
                                                   const uint16_t* __restrict__ U, int ldu,
                                                   const uint16_t* __restrict__ V, int ldv,
                                                   int m, int n, float* __restrict__ grad,
                                                   long long gstride, int add) {
    using namespace seg;
    __shared__ __align__(128) uint8_t sU[2][WG_ROWS * 128];
    __shared__ __align__(128) uint8_t sV[2][WG_ROWS * 256];
    const int sg = blockIdx.z;
    const int r0 = sr.r0[sg], r1 = sr.r1[sg];
    const int m0 = blockIdx.y * WG_BM, n0 = blockIdx.x * WG_BN;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int wm = warp & 1, wn = warp >> 1;
    const uint32_t ua = smem_u32(sU), va = smem_u32(sV);
    const int nsteps = (r1 - r0 + WG_ROWS - 1) / WG_ROWS;
    auto load = [&](int st, int buf) {
        const int rb = r0 + st * WG_ROWS;
        for (int i = tid; i < WG_ROWS * 8; i += 128) {  // U: 32 rows x 8 units (64 m)
            const int r = i >> 3, u = i & 7;
            const bool ok = rb + r < r1;
            cp_async16(ua + buf * WG_ROWS * 128 + r * 128 + ((u ^ (r & 7)) << 4),
                       U + (size_t)(ok ? rb + r : r0) * ldu + m0 + u * 8, ok);
        }
        for (int i = tid; i < WG_ROWS * 16; i += 128) {  // V: 32 rows x 16 units (128 n)
            const int r = i >> 4, u = i & 15;
            const bool ok = rb + r < r1;
            cp_async16(va + buf * WG_ROWS * 256 + r * 256 + ((u ^ (r & 7)) << 4),
                       V + (size_t)(ok ? rb + r : r0) * ldv + n0 + u * 8, ok);
        }
    };
    float acc[2][8][4];
#pragma unroll
    for (int i = 0; i < 2; ++i)
#pragma unroll
        for (int j = 0; j < 8; ++j) acc[i][j][0] = acc[i][j][1] = acc[i][j][2] = acc[i][j][3] = 0.f;
    const int mi = lane >> 3, rr = lane & 7;
    if (nsteps > 0) load(0, 0);
    cp_async_commit();
    for (int st = 0; st < nsteps; ++st) {
        const int buf = st & 1;
        if (st + 1 < nsteps) load(st + 1, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t ub = ua + buf * WG_ROWS * 128, vb = va + buf * WG_ROWS * 256;
#pragma unroll
        for (int ks = 0; ks < 2; ++ks) {
            // A = U^T: transposed 8x8 blocks of U (rows = k, columns = m)
            uint32_t a[2][4];
#pragma unroll
            for (int mt = 0; mt < 2; ++mt) {
                const int r = ks * 16 + rr + 8 * (mi >> 1);
                const int u = wm * 4 + mt * 2 + (mi & 1);
                ldsm_x4_t(ub + r * 128 + ((u ^ (r & 7)) << 4), a[mt][0], a[mt][1], a[mt][2],
                          a[mt][3]);
            }
#pragma unroll
            for (int nb = 0; nb < 4; ++nb) {
                const int r = ks * 16 + rr + 8 * (mi & 1), u = wn * 8 + nb * 2 + (mi >> 1);
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vb + r * 256 + ((u ^ (r & 7)) << 4), b0, b1, b2, b3);
#pragma unroll
                for (int mt = 0; mt < 2; ++mt) {
                    mma_bf16(acc[mt][2 * nb], a[mt][0], a[mt][1], a[mt][2], a[mt][3], b0, b1);
                    mma_bf16(acc[mt][2 * nb + 1], a[mt][0], a[mt][1], a[mt][2], a[mt][3], b2, b3);
                }
            }
        }
        __syncthreads();
    }
    const int g = lane >> 2, q = lane & 3;
    float* gt = grad + (size_t)sr.tenant[sg] * gstride;
#pragma unroll
    for (int mt = 0; mt < 2; ++mt)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int row = m0 + wm * 32 + mt * 16 + g + 8 * h;
            float* o = gt + (size_t)row * n + n0 + wn * 64 + 2 * q;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                float2 v = make_float2(acc[mt][j][2 * h], acc[mt][j][2 * h + 1]);
                if (add) {
                    const float2 old = *reinterpret_cast<const float2*>(o + j * 8);
                    v.x += old.x;
                    v.y += old.y;
                }
                *reinterpret_cast<float2*>(o + j * 8) = v;
            }
        }
}

jnx_status seg_wgrad_launch(const SegRows& sr, const uint16_t* U, int ldu, const uint16_t* V,
                            int ldv, int m, int n, float* grad, long long gstride, bool add,
                            cudaStream_t s) {
    if (m % seg::WG_BM || n % seg::WG_BN || ldu % 8 || ldv % 8)
        return fail(JNX_ERR_UNSUPPORTED, "weight gradient: %d x %d", m, n);
    if (sr.n <= 0) return JNX_OK;
    if (m / seg::WG_BM > 65535 || sr.n > 65535)
        return fail(JNX_ERR_UNSUPPORTED, "weight gradient: grid too large");
    k_seg_wgrad<<<dim3(n / seg::WG_BN, m / seg::WG_BM, sr.n), 128, 0, s>>>(sr, U, ldu, V, ldv, m,
                                                                          n, grad, gstride,
                                                                          add ? 1 : 0);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "weight gradient: %s", cudaGetErrorString(e));
}

// ---------------------------------------------------------------------------
// MLP heads: d hidden[row] = (dz[s] W1) / L_s for every row of sample s.
// One CTA per (sample, 256-column block); dz [n_samples, ldz] fp32.
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(256) k_mlp_dfeat(const float* __restrict__ dz, int ldz,
                                                   const int* __restrict__ cu,
                                                   const int* __restrict__ sample_slot,
                                                   const __grid_constant__ MlpFeatTable tab, int d,
                                                   float* __restrict__ dh) {
    const int s = blockIdx.x;
    const int c = blockIdx.y * 256 + threadIdx.x;
    const int slot = sample_slot[s];
    const uint16_t* w1 = tab.w1[slot];
    const int hid = tab.hid[slot];
    if (w1 == nullptr || c >= d) return;  // not an MLP slot
    float acc = 0.f;
    for (int j = 0; j < hid; ++j) acc += dz[(size_t)s * ldz + j] * bf2f(w1[(size_t)j * d + c]);
    const int r0 = cu[s], r1 = cu[s + 1];
    const float v = acc / (float)(r1 - r0);
    for (int r = r0; r < r1; ++r) dh[(size_t)r * d + c] = v;
}

jnx_status mlp_dfeat_launch(const float* dz, int ldz, const int* cu, const int* sample_slot,
                            int n_samples, const MlpFeatTable& tab, int d, float* dh,
                            cudaStream_t s) {
    if (n_samples <= 0) return JNX_OK;
    k_mlp_dfeat<<<dim3(n_samples, (d + 255) / 256), 256, 0, s>>>(dz, ldz, cu, sample_slot, tab, d,
                                                                dh);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "MLP feature gradient: %s", cudaGetErrorString(e));
}

// fp32 -> bf16 of a [rows, cols] block with row strides (the query heads'
// dk | dv rows into one bf16 operand).
__global__ void __launch_bounds__(256) k_to_bf16(const float* __restrict__ src, int lds, int rows,
                                                 int cols, uint16_t* __restrict__ dst, int ldd) {
    const long long i = (long long)blockIdx.x * 256 + threadIdx.x;
    if (i >= (long long)rows * (cols / 2)) return;
    const int r = (int)(i / (cols / 2)), c = (int)(i % (cols / 2)) * 2;
    const float2 v = *reinterpret_cast<const float2*>(src + (size_t)r * lds + c);
    *reinterpret_cast<uint32_t*>(dst + (size_t)r * ldd + c) = pack_bf2(v.x, v.y);
}

jnx_status to_bf16_launch(const float* src, int lds, int rows, int cols, uint16_t* dst, int ldd,
                          cudaStream_t s) {
    if (cols % 2 || lds % 2 || ldd % 2) return fail(JNX_ERR_UNSUPPORTED, "to bf16: odd widths");
    const long long n = (long long)rows * (cols / 2);
    if (n <= 0) return JNX_OK;
    k_to_bf16<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(src, lds, rows, cols, dst, ldd);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "to bf16: %s", cudaGetErrorString(e));
}

}  // namespace jnx
