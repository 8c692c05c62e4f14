// Varlen attention confined to each sample (block-diagonal, bidirectional).
//
// Every sample is one observation prefix; its tokens attend to each other
// and to nothing else, so the grid only visits (sample, 64-query tile, head)
// triples inside a sample and the key loop only walks that sample's keys:
// no cross-sample tile is ever computed.  Tiles start at the sample's first
// token, so a sample's result is the same wherever it sits in the packed
// batch (grouped == isolated).
//
// Two kernels, chosen per head dim in attention_launch:
//  k_attn     flash-style online softmax in fp32 with bf16 mma.sync
//             (m16n8k16): each of the 4 warps owns 16 query rows; K/V tiles
//             stream through a double-buffered cp.async ring in XOR-swizzled
//             shared memory read with ldmatrix;
//  k_attn_tc  the same algorithm on tcgen05: S and O accumulate in TMEM, Q/K/V
//             arrive by TMA, P goes through shared memory (see below).
// Q, K, V come from the fused projection output [N, (H + 2 Hkv) hd]; query
// head h reads K/V head h / (H / Hkv) (MQA when Hkv = 1).
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

namespace attn {
constexpr int BM = 64;  // query rows per CTA (16 per warp)
}

// byte offset of 16-byte chunk `ch` of row `r` in a [rows][HD] bf16 tile
template <int HD>
__device__ __forceinline__ uint32_t sw_off(int r, int ch) {
    return (uint32_t)(r * HD * 2 + ((ch ^ (r & 7)) << 4));
}

template <int HD, int BN>
__global__ void __launch_bounds__(128) k_attn(const uint16_t* __restrict__ qkv, int ldq, int H,
                                              int Hkv, const int* __restrict__ cu,
                                              int tiles_per_sample, float scale_log2,
                                              uint16_t* __restrict__ out, int ldo) {
    using attn::BM;
    constexpr int CH = HD / 8;   // 16-byte chunks per row
    constexpr int NT = BN / 8;   // S n-tiles per warp
    constexpr int OT = HD / 8;   // O n-tiles per warp
    extern __shared__ __align__(128) uint8_t sm[];
    uint8_t* sQ = sm;
    uint8_t* sK = sQ + BM * HD * 2;
    uint8_t* sV = sK + 2 * BN * HD * 2;

    const int s = blockIdx.x / tiles_per_sample;
    const int qt = blockIdx.x % tiles_per_sample;
    const int h = blockIdx.y;
    const int kvh = h / (H / Hkv);
    const int start = cu[s];
    const int L = cu[s + 1] - start;
    const int q0 = qt * BM;
    if (q0 >= L) return;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint16_t* Qg = qkv + (size_t)start * ldq + h * HD;
    const uint16_t* Kg = qkv + (size_t)start * ldq + (H + kvh) * HD;
    const uint16_t* Vg = qkv + (size_t)start * ldq + (H + Hkv + kvh) * HD;

    const uint32_t sQa = smem_u32(sQ), sKa = smem_u32(sK), sVa = smem_u32(sV);

    // Q tile (rows beyond the sample are zero)
    for (int i = tid; i < BM * CH; i += 128) {
        const int r = i / CH, ch = i % CH;
        const bool ok = q0 + r < L;
        cp_async16(sQa + sw_off<HD>(r, ch), ok ? (const void*)(Qg + (size_t)(q0 + r) * ldq + ch * 8)
                                               : (const void*)qkv,
                   ok);
    }
    auto load_kv = [&](int kt, int buf) {
        const int k0 = kt * BN;
        for (int i = tid; i < BN * CH; i += 128) {
            const int r = i / CH, ch = i % CH;
            const bool ok = k0 + r < L;
            const size_t off = (size_t)(k0 + r) * ldq + ch * 8;
            cp_async16(sKa + buf * BN * HD * 2 + sw_off<HD>(r, ch),
                       ok ? (const void*)(Kg + off) : (const void*)qkv, ok);
            cp_async16(sVa + buf * BN * HD * 2 + sw_off<HD>(r, ch),
                       ok ? (const void*)(Vg + off) : (const void*)qkv, ok);
        }
    };
    const int n_kt = (L + BN - 1) / BN;
    load_kv(0, 0);
    cp_async_commit();

    float o[OT][4];
#pragma unroll
    for (int i = 0; i < OT; ++i) o[i][0] = o[i][1] = o[i][2] = o[i][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;

    const int g = lane >> 2, t = lane & 3;
    const int mi = lane >> 3, rr = lane & 7;
    const int qrow = warp * 16;

    for (int kt = 0; kt < n_kt; ++kt) {
        const int buf = kt & 1;
        if (kt + 1 < n_kt) load_kv(kt + 1, buf ^ 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();

        const uint32_t kb = sKa + buf * BN * HD * 2;
        const uint32_t vb = sVa + buf * BN * HD * 2;

        // S = Q K^T (16 x BN per warp)
        float sc[NT][4];
#pragma unroll
        for (int i = 0; i < NT; ++i) sc[i][0] = sc[i][1] = sc[i][2] = sc[i][3] = 0.f;
#pragma unroll
        for (int ks = 0; ks < HD / 16; ++ks) {
            uint32_t a0, a1, a2, a3;
            ldsm_x4(sQa + sw_off<HD>(qrow + rr + 8 * (mi & 1), ks * 2 + (mi >> 1)), a0, a1, a2, a3);
#pragma unroll
            for (int nb = 0; nb < BN / 16; ++nb) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4(kb + sw_off<HD>(nb * 16 + rr + 8 * (mi >> 1), ks * 2 + (mi & 1)), b0, b1,
                        b2, b3);
                mma_bf16(sc[2 * nb], a0, a1, a2, a3, b0, b1);
                mma_bf16(sc[2 * nb + 1], a0, a1, a2, a3, b2, b3);
            }
        }

        // scale to log2 domain, mask keys past the sample, online softmax
        const int kbase = kt * BN;
        float mx0 = m0, mx1 = m1;
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            const int key = kbase + i * 8 + 2 * t;
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const bool ok = key + (e & 1) < L;
                sc[i][e] = ok ? sc[i][e] * scale_log2 : -INFINITY;
            }
            mx0 = fmaxf(mx0, fmaxf(sc[i][0], sc[i][1]));
            mx1 = fmaxf(mx1, fmaxf(sc[i][2], sc[i][3]));
        }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        const float al0 = exp2f(m0 - mx0), al1 = exp2f(m1 - mx1);
        m0 = mx0;
        m1 = mx1;
        float rs0 = 0.f, rs1 = 0.f;
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            sc[i][0] = exp2f(sc[i][0] - m0);
            sc[i][1] = exp2f(sc[i][1] - m0);
            sc[i][2] = exp2f(sc[i][2] - m1);
            sc[i][3] = exp2f(sc[i][3] - m1);
            rs0 += sc[i][0] + sc[i][1];
            rs1 += sc[i][2] + sc[i][3];
        }
        l0 = l0 * al0 + rs0;
        l1 = l1 * al1 + rs1;
#pragma unroll
        for (int i = 0; i < OT; ++i) {
            o[i][0] *= al0;
            o[i][1] *= al0;
            o[i][2] *= al1;
            o[i][3] *= al1;
        }

        // O += P V
#pragma unroll
        for (int kk = 0; kk < BN / 16; ++kk) {
            const uint32_t a0 = pack_bf2(sc[2 * kk][0], sc[2 * kk][1]);
            const uint32_t a1 = pack_bf2(sc[2 * kk][2], sc[2 * kk][3]);
            const uint32_t a2 = pack_bf2(sc[2 * kk + 1][0], sc[2 * kk + 1][1]);
            const uint32_t a3 = pack_bf2(sc[2 * kk + 1][2], sc[2 * kk + 1][3]);
#pragma unroll
            for (int np = 0; np < HD / 16; ++np) {
                uint32_t b0, b1, b2, b3;
                ldsm_x4_t(vb + sw_off<HD>(kk * 16 + rr + 8 * (mi & 1), 2 * np + (mi >> 1)), b0, b1,
                          b2, b3);
                mma_bf16(o[2 * np], a0, a1, a2, a3, b0, b1);
                mma_bf16(o[2 * np + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        __syncthreads();
    }

    l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
    const float i0 = 1.f / l0, i1 = 1.f / l1;
    const int r0 = q0 + qrow + g, r1 = r0 + 8;
    uint16_t* ob = out + (size_t)start * ldo + h * HD;
#pragma unroll
    for (int i = 0; i < OT; ++i) {
        const int col = i * 8 + 2 * t;
        if (r0 < L)
            *reinterpret_cast<uint32_t*>(ob + (size_t)r0 * ldo + col) =
                pack_bf2(o[i][0] * i0, o[i][1] * i0);
        if (r1 < L)
            *reinterpret_cast<uint32_t*>(ob + (size_t)r1 * ldo + col) =
                pack_bf2(o[i][2] * i1, o[i][3] * i1);
    }
}

// ---------------------------------------------------------------------------
// tcgen05 version.  One CTA = (sample, 128-query tile, head), 128 threads:
// thread r owns query row r for the softmax and the epilogue; thread 0 also
// issues the TMA copies and the MMAs.  Per key tile of BN keys:
//   S = Q K^T          tcgen05.mma (M=128, N=BN, K=HD) into TMEM
//   softmax            each thread reads its S row from TMEM twice (row max,
//                      then p = 2^(s*scale*log2e - m)), rescales its O row in
//                      TMEM when the running max moved, and writes p as bf16
//                      into shared memory in the 128-byte-swizzled K-major
//                      layout the next MMA reads
//   O += P V           tcgen05.mma (M=128, N=HD, K=BN), V read MN-major
// K/V tiles are double-buffered: the copy of tile kt+1 runs during tile kt.
// The commit that follows S(kt) also covers PV(kt-1), so one barrier wait
// tells the softmax threads that O, P and the older K/V buffer are free.
// ---------------------------------------------------------------------------
namespace attn_tc {
constexpr int BM = 128;
}

template <int HD, int BN>
struct AttnTcCfg {
    // P rows are 128 bytes (64 keys) in the 128-byte-swizzled layout the PV
    // MMA reads, so a key tile narrower than 64 would not fill its buffer.
    static_assert(BN == 64 || BN == 128, "key tile must be 64 or 128 keys");
    static_assert(HD % 64 == 0 && HD <= 256, "head dim must be 64, 128 or 256");
    static constexpr int QB = attn_tc::BM * HD * 2;  // Q tile bytes
    static constexpr int KB = BN * HD * 2;           // K (or V) tile bytes
    static constexpr int PB = attn_tc::BM * BN * 2;  // P tile bytes
    static constexpr int SMEM = QB + 4 * KB + PB + 1024 + 256;
    static constexpr uint32_t O_COL = 128;           // TMEM column of the O accumulator
    static constexpr uint32_t TCOLS = O_COL + HD <= 256 ? 256 : 512;  // TMEM columns held
};

template <int HD, int BN>
__global__ void __launch_bounds__(128, 1)
    k_attn_tc(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tkv,
              const int* __restrict__ cu, int tiles_per_sample, int H, int Hkv, float scale_log2,
              uint16_t* __restrict__ out, int ldo, int* status) {
    using C = AttnTcCfg<HD, BN>;
    constexpr int BM = attn_tc::BM;
    constexpr int NCH = HD / 64;  // 64-column chunks of a head row
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* sQ = sm;
    // K/V buffer b: K at QB + 2b KB, V right after it
    auto sK = [&](int b) { return sm + C::QB + 2 * b * C::KB; };
    auto sV = [&](int b) { return sm + C::QB + (2 * b + 1) * C::KB; };
    uint8_t* sP = sm + C::QB + 4 * C::KB;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sP + C::PB);
    uint64_t* q_full = bars;
    uint64_t* kv_full = bars + 1;  // [2]
    uint64_t* s_full = bars + 3;
    uint64_t* pv_done = bars + 4;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 5);

    const int s = blockIdx.x / tiles_per_sample;
    const int qt = blockIdx.x % tiles_per_sample;
    const int h = blockIdx.y;
    const int kvh = h / (H / Hkv);
    const int start = cu[s];
    const int L = cu[s + 1] - start;
    const int q0 = qt * BM;
    if (q0 >= L) return;  // uniform for the whole CTA

    const int tid = threadIdx.x, warp = tid >> 5;
    if (tid == 0) {
        mbar_init(q_full, 1);
        mbar_init(&kv_full[0], 1);
        mbar_init(&kv_full[1], 1);
        mbar_init(s_full, 1);
        mbar_init(pv_done, 1);
        fence_barrier_init();
        fence_proxy_async();
    }
    if (warp == 0) {
        tmem_alloc(tmem_slot, C::TCOLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
    const uint32_t tS = tbase + lane_base;
    const uint32_t tO = tbase + lane_base + C::O_COL;
    const int n_kt = (L + BN - 1) / BN;
    bool ok = true;

    auto issue_kv = [&](int kt, int buf) {
        mbar_arrive_expect_tx(&kv_full[buf], 2 * C::KB);
        const int y = start + kt * BN;
#pragma unroll
        for (int c = 0; c < NCH; ++c) {
            tma_load_2d(sK(buf) + c * BN * 128, &tkv, (H + kvh) * HD + c * 64, y, &kv_full[buf]);
            tma_load_2d(sV(buf) + c * BN * 128, &tkv, (H + Hkv + kvh) * HD + c * 64, y,
                        &kv_full[buf]);
        }
    };
    if (tid == 0) {
        mbar_arrive_expect_tx(q_full, C::QB);
#pragma unroll
        for (int c = 0; c < NCH; ++c)
            tma_load_2d(sQ + c * BM * 128, &tq, h * HD + c * 64, start + q0, q_full);
        issue_kv(0, 0);
    }

    constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
    constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, HD) | (1u << 16);  // B (V) MN-major
    float m = -INFINITY, l = 0.f;

    for (int kt = 0; kt < n_kt; ++kt) {
        const int buf = kt & 1;
        if (tid == 0) {
            if (kt == 0) ok = ok && mbar_wait(q_full, 0);
            ok = ok && mbar_wait(&kv_full[buf], (kt >> 1) & 1);
            tc_fence_after();
            const uint32_t qa = smem_u32(sQ), ka = smem_u32(sK(buf));
#pragma unroll
            for (int ks = 0; ks < HD / 16; ++ks)
                tc_mma_f16(tS - lane_base, sw128_desc(qa + (ks >> 2) * BM * 128 + (ks & 3) * 32),
                           sw128_desc(ka + (ks >> 2) * BN * 128 + (ks & 3) * 32), IDESC_S,
                           ks > 0);
            tc_commit(s_full);
        }
        __syncwarp();
        ok = mbar_wait(s_full, kt & 1) && ok;
        tc_fence_after();
        if (tid == 0 && kt + 1 < n_kt) issue_kv(kt + 1, buf ^ 1);  // PV(kt-1) is done

        // pass 1: row max over this tile's valid keys
        const int kbase = kt * BN;
        float mx = -INFINITY;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(tS + c * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int e = 0; e < 32; ++e)
                if (kbase + c * 32 + e < L) mx = fmaxf(mx, __uint_as_float(r[e]) * scale_log2);
        }
        const float m_new = fmaxf(m, mx);
        const float alpha = exp2f(m - m_new);
        if (kt > 0 && __any_sync(0xffffffffu, alpha < 1.0f)) {
#pragma unroll 1
            for (int c = 0; c < HD / 32; ++c) {
                uint32_t r[32];
                tmem_ld32(tO + c * 32, r);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(__uint_as_float(r[e]) * alpha);
                tmem_st32(tO + c * 32, r);
            }
            tmem_st_wait();
        }
        m = m_new;
        // pass 2: p = 2^(s * scale - m) -> bf16 P in smem, row sum
        float rs = 0.f;
#pragma unroll 1
        for (int c = 0; c < BN / 32; ++c) {
            uint32_t r[32];
            tmem_ld32(tS + c * 32, r);
            tmem_ld_wait();
            float p[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                p[e] = (kbase + c * 32 + e < L) ? exp2f(__uint_as_float(r[e]) * scale_log2 - m)
                                                : 0.f;
                rs += p[e];
            }
            // keys c*32 .. c*32+31 = 16-byte units 4(c%2) .. 4(c%2)+3 of chunk c/2
            uint8_t* prow = sP + (c >> 1) * BM * 128 + tid * 128;
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int unit = 4 * (c & 1) + u;
                uint4 w;
                w.x = pack_bf2(p[8 * u + 0], p[8 * u + 1]);
                w.y = pack_bf2(p[8 * u + 2], p[8 * u + 3]);
                w.z = pack_bf2(p[8 * u + 4], p[8 * u + 5]);
                w.w = pack_bf2(p[8 * u + 6], p[8 * u + 7]);
                *reinterpret_cast<uint4*>(prow + ((unit ^ (tid & 7)) << 4)) = w;
            }
        }
        l = l * alpha + rs;
        fence_proxy_async();
        tc_fence_before();
        __syncthreads();
        if (tid == 0) {
            tc_fence_after();
            const uint32_t pa = smem_u32(sP), va = smem_u32(sV(buf));
#pragma unroll
            for (int ks = 0; ks < BN / 16; ++ks)
                tc_mma_f16(tO - lane_base,
                           sw128_desc(pa + (ks >> 2) * BM * 128 + (ks & 3) * 32),
                           sw128_desc_mn(va + ks * 16 * 128, BN * 128, 1024), IDESC_PV,
                           (kt > 0 || ks > 0));
            if (kt == n_kt - 1) tc_commit(pv_done);
        }
        __syncwarp();
    }
    ok = mbar_wait(pv_done, 0) && ok;
    tc_fence_after();
    if (!ok && tid == 0) report(status, JNX_ERR_TIMEOUT);

    // epilogue: O / l -> bf16
    const float inv = 1.0f / l;
    const int row = q0 + tid;
    uint16_t* orow = out + (size_t)(start + row) * ldo + h * HD;
#pragma unroll 1
    for (int c = 0; c < HD / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tO + c * 32, r);
        tmem_ld_wait();
        if (row < L) {
            uint4* dst = reinterpret_cast<uint4*>(orow + c * 32);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                uint4 w;
                w.x = pack_bf2(__uint_as_float(r[8 * v + 0]) * inv, __uint_as_float(r[8 * v + 1]) * inv);
                w.y = pack_bf2(__uint_as_float(r[8 * v + 2]) * inv, __uint_as_float(r[8 * v + 3]) * inv);
                w.z = pack_bf2(__uint_as_float(r[8 * v + 4]) * inv, __uint_as_float(r[8 * v + 5]) * inv);
                w.w = pack_bf2(__uint_as_float(r[8 * v + 6]) * inv, __uint_as_float(r[8 * v + 7]) * inv);
                dst[v] = w;
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tbase, C::TCOLS);
}

template <int HD, int BN>
static jnx_status launch_attn_tc(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv,
                                 const int* cu, int S, int max_seqlen, uint16_t* out, int ldo,
                                 int* status, cudaStream_t s) {
    using C = AttnTcCfg<HD, BN>;
    static bool attr = false;
    if (!attr) {
        if (cudaFuncSetAttribute(k_attn_tc<HD, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 C::SMEM) != cudaSuccess)
            return fail(JNX_ERR_CUDA, "attention: smem attribute");
        attr = true;
    }
    CUtensorMap tq, tkv;
    if (!make_tmap_bf16(&tq, qkv, n_tokens, ldq, ldq, attn_tc::BM, 64) ||
        !make_tmap_bf16(&tkv, qkv, n_tokens, ldq, ldq, BN, 64))
        return fail(JNX_ERR_CUDA, "attention: tensor map encode failed");
    const int tps = (max_seqlen + attn_tc::BM - 1) / attn_tc::BM;
    const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
    dim3 grid(S * tps, H);
    k_attn_tc<HD, BN><<<grid, 128, C::SMEM, s>>>(tq, tkv, cu, tps, H, Hkv, scale_log2, out, ldo,
                                                 status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
}

template <int HD, int BN>
static cudaError_t launch_attn(const uint16_t* qkv, int ldq, int H, int Hkv, const int* cu, int S,
                               int max_seqlen, uint16_t* out, int ldo, cudaStream_t s) {
    constexpr int smem = attn::BM * HD * 2 + 4 * BN * HD * 2;
    static bool attr = false;
    if (!attr) {
        cudaError_t e =
            cudaFuncSetAttribute(k_attn<HD, BN>, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
        if (e != cudaSuccess) return e;
        attr = true;
    }
    const int tps = (max_seqlen + attn::BM - 1) / attn::BM;
    const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
    dim3 grid(S * tps, H);
    k_attn<HD, BN><<<grid, 128, smem, s>>>(qkv, ldq, H, Hkv, cu, tps, scale_log2, out, ldo);
    return cudaGetLastError();
}

jnx_status attention_launch(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv, int hd,
                            const int* cu, int S, int max_seqlen, uint16_t* out, int ldo,
                            int* status, cudaStream_t s) {
    if (S == 0 || max_seqlen == 0) return JNX_OK;
    if (Hkv <= 0 || H % Hkv) return fail(JNX_ERR_UNSUPPORTED, "attention: H %% Hkv != 0");
    if ((long long)S * ((max_seqlen + attn::BM - 1) / attn::BM) > 0x7FFFFFFFLL || H > 65535)
        return fail(JNX_ERR_UNSUPPORTED, "attention: grid too large");
    // Per head dim, the faster of the two kernels as measured on GB300 for
    // prefixes of 260..840 tokens: the mma.sync kernel for 64 / 128 (181 /
    // 224 TFLOP/s against 71 / 143 for this tcgen05 version, whose single
    // 128-thread CTA per SM leaves the per-tile copy and softmax latencies
    // exposed), the tcgen05 kernel for 256 (300 against 281).
    cudaError_t e = cudaSuccess;
    switch (hd) {
        case 64:
            e = launch_attn<64, 64>(qkv, ldq, H, Hkv, cu, S, max_seqlen, out, ldo, s);
            return e == cudaSuccess ? JNX_OK
                                    : fail(JNX_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
        case 128:
            e = launch_attn<128, 64>(qkv, ldq, H, Hkv, cu, S, max_seqlen, out, ldo, s);
            return e == cudaSuccess ? JNX_OK
                                    : fail(JNX_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
        case 256:
            return launch_attn_tc<256, 64>(qkv, ldq, n_tokens, H, Hkv, cu, S, max_seqlen, out,
                                           ldo, status, s);
        default:
            return fail(JNX_ERR_UNSUPPORTED, "attention: head_dim %d not in {64,128,256}", hd);
    }
}

}  // namespace jnx
