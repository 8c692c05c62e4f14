// Per-tenant LoRA on the backbone projections (the skewed 64-tenant
// workload): y += (x A_t^T) B_t^T for the rows of tenant t, rank r = 16.
//
// The low-rank update is split in two:
//   down  t = x A_t^T  [rows, parts * r] bf16   -- this file: a segmented
//         mma.sync kernel whose 64-row tiles never straddle two tenants
//         (tiles start at each tenant's first row), so each tile applies one
//         tenant's A;
//   up    t B_t^T is one more K = 16 tcgen05 MMA into the projection GEMM's
//         accumulator (gemm.cu, gemm_launch_lora), before RoPE for Q/K/V and
//         before the residual add for O; that GEMM lays its tiles out per
//         tenant segment too.
// Rows of one tenant are contiguous because the plan packs tenant by tenant.
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

namespace lora {
constexpr int BM = 64, BK = 64;
}

template <int HD>
__device__ __forceinline__ uint32_t lsw(int r, int ch) {
    return (uint32_t)(r * HD * 2 + ((ch ^ (r & 7)) << 4));
}

// t[row, p*r + j] = sum_k x[row, k] A_p[tenant][j, k] for the parts p < NP.
// One CTA per (tenant segment, 64-row tile); 4 warps x 16 rows; NP*r output
// columns per row (NT = NP*r/8 mma n-tiles per warp).
template <int NP>
__global__ void __launch_bounds__(128) k_lora_down(const uint16_t* __restrict__ x, int ldx, int K,
                                                   const __grid_constant__ LoraSlots ls,
                                                   const __grid_constant__ LoraDown ld,
                                                   uint16_t* __restrict__ t, int ldt) {
    using lora::BK;
    using lora::BM;
    constexpr int R = kLoraRank;
    constexpr int NO = NP * R;   // output columns
    constexpr int NT = NO / 8;   // mma n-tiles
    __shared__ __align__(128) uint8_t sX[2][BM * BK * 2];
    __shared__ __align__(128) uint8_t sA[2][NO * BK * 2];

    // which tenant segment / tile
    int seg = 0;
    while (seg + 1 < ls.n && ls.tile_start[seg + 1] <= (int)blockIdx.x) ++seg;
    const int r0 = ls.r0[seg], r1 = ls.r1[seg];
    const int row0 = r0 + ((int)blockIdx.x - ls.tile_start[seg]) * BM;
    if (row0 >= r1) return;
    const int tenant = ls.tenant[seg];
    const uint16_t* Ap[NP];
#pragma unroll
    for (int p = 0; p < NP; ++p) Ap[p] = ld.a[p] + (size_t)tenant * R * K;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t xa = smem_u32(sX), aa = smem_u32(sA);
    auto load = [&](int kb, int buf) {
        const int k0 = kb * BK;
        for (int i = tid; i < BM * 8; i += 128) {
            const int r = i / 8, ch = i % 8;
            const bool ok = row0 + r < r1;
            cp_async16(xa + buf * BM * BK * 2 + lsw<BK>(r, ch),
                       ok ? (const void*)(x + (size_t)(row0 + r) * ldx + k0 + ch * 8)
                          : (const void*)x,
                       ok);
        }
        for (int i = tid; i < NO * 8; i += 128) {
            const int r = i / 8, ch = i % 8;
            cp_async16(aa + buf * NO * BK * 2 + lsw<BK>(r, ch),
                       Ap[r / R] + (size_t)(r % R) * K + k0 + ch * 8, true);
        }
    };
    float acc[NT][4];
#pragma unroll
    for (int i = 0; i < NT; ++i) acc[i][0] = acc[i][1] = acc[i][2] = acc[i][3] = 0.f;
    const int nkb = K / BK;
    const int mi = lane >> 3, rr = lane & 7;
    load(0, 0);
    cp_async_commit();
    for (int kb = 0; kb < nkb; ++kb) {
        const int buf = kb & 1;
        if (kb + 1 < nkb) load(kb + 1, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t xb = xa + buf * BM * BK * 2, ab = aa + buf * NO * BK * 2;
#pragma unroll
        for (int ks = 0; ks < BK / 16; ++ks) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(xb + lsw<BK>(warp * 16 + rr + 8 * (mi & 1), ks * 2 + (mi >> 1)), a0, a1, a2,
                    a3);
#pragma unroll
            for (int nb = 0; nb < NT / 2; ++nb) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(ab + lsw<BK>(nb * 16 + rr + 8 * (mi >> 1), ks * 2 + (mi & 1)), b0, b1, b2,
                        b3);
                mma_bf16(acc[2 * nb], a0, a1, a2, a3, b0, b1);
                mma_bf16(acc[2 * nb + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        __syncthreads();
    }
    const int g = lane >> 2, tq = lane & 3;
    const int ra = row0 + warp * 16 + g, rb = ra + 8;
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int col = i * 8 + 2 * tq;
        if (ra < r1)
            *reinterpret_cast<uint32_t*>(t + (size_t)ra * ldt + col) = pack_bf2(acc[i][0], acc[i][1]);
        if (rb < r1)
            *reinterpret_cast<uint32_t*>(t + (size_t)rb * ldt + col) = pack_bf2(acc[i][2], acc[i][3]);
    }
}

jnx_status lora_down_launch(const jnx_group* g, const uint16_t* x, int ldx, int K, int n_parts,
                            const uint16_t* const* a, uint16_t* t, int ldt, cudaStream_t s) {
    if (K % lora::BK) return fail(JNX_ERR_UNSUPPORTED, "lora: K %% 64 != 0");
    LoraDown ld{};
    for (int p = 0; p < n_parts; ++p) ld.a[p] = a[p];
    for (int g0 = 0; g0 < g->n_slots; g0 += kLoraMaxSlots) {
        LoraSlots ls{};
        ls.g0 = g0;
        ls.n = g->n_slots - g0 < kLoraMaxSlots ? g->n_slots - g0 : kLoraMaxSlots;
        int tiles = 0;
        for (int i = 0; i < ls.n; ++i) {
            ls.tenant[i] = g->h_slot_tenant[g0 + i];
            ls.r0[i] = g->h_cu_seqlens[g->h_seg_offsets[g0 + i]];
            ls.r1[i] = g->h_cu_seqlens[g->h_seg_offsets[g0 + i + 1]];
            ls.tile_start[i] = tiles;
            tiles += (ls.r1[i] - ls.r0[i] + lora::BM - 1) / lora::BM;
        }
        if (tiles == 0) continue;
        if (n_parts == 3)
            k_lora_down<3><<<tiles, 128, 0, s>>>(x, ldx, K, ls, ld, t, ldt);
        else
            k_lora_down<1><<<tiles, 128, 0, s>>>(x, ldx, K, ls, ld, t, ldt);
    }
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "lora down: %s", cudaGetErrorString(e));
}

}  // namespace jnx
