// Varlen attention confined to each sample (block-diagonal, bidirectional).
//
// Every sample is one observation prefix; its tokens attend to each other
// and to nothing else, so the grid only visits (sample, 64-query tile, head)
// triples inside a sample and the key loop only walks that sample's keys:
// no cross-sample tile is ever computed.  Tiles start at the sample's first
// token, so a sample's result is the same wherever it sits in the packed
// batch (grouped == isolated).
//
// Flash-style online softmax in fp32 with bf16 mma.sync (m16n8k16): each of
// the 4 warps owns 16 query rows; K/V tiles stream through a double-buffered
// cp.async ring in XOR-swizzled shared memory read with ldmatrix.  Q, K, V
// come from the fused projection output [N, (H + 2 Hkv) hd]; query head h
// reads K/V head h / (H / Hkv) (MQA when Hkv = 1).
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

jnx_status attention_launch(const uint16_t* qkv, int ldq, int H, int Hkv, int hd, const int* cu,
                            int S, int max_seqlen, uint16_t* out, int ldo, cudaStream_t s) {
    if (S == 0 || max_seqlen == 0) return JNX_OK;
    if (Hkv <= 0 || H % Hkv) return fail(JNX_ERR_UNSUPPORTED, "attention: H %% Hkv != 0");
    if ((long long)S * ((max_seqlen + attn::BM - 1) / attn::BM) > 0x7FFFFFFFLL || H > 65535)
        return fail(JNX_ERR_UNSUPPORTED, "attention: grid too large");
    cudaError_t e;
    switch (hd) {
        case 64: e = launch_attn<64, 64>(qkv, ldq, H, Hkv, cu, S, max_seqlen, out, ldo, s); break;
        case 128: e = launch_attn<128, 64>(qkv, ldq, H, Hkv, cu, S, max_seqlen, out, ldo, s); break;
        case 256: e = launch_attn<256, 32>(qkv, ldq, H, Hkv, cu, S, max_seqlen, out, ldo, s); break;
        default: return fail(JNX_ERR_UNSUPPORTED, "attention: head_dim %d not in {64,128,256}", hd);
    }
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
}

}  // namespace jnx
