// Dense bf16 GEMM on the 5th-generation tensor cores (tcgen05, sm_103a).
//
//   C[M, N] = A[M, K] . B[N, K]^T      (A = activations, B = weights [out, in])
//
// One persistent CTA per SM walks output tiles of 128 x 256.  Warp roles:
//   warp 0     TMA producer: 128x64 A and 256x64 B boxes (128-byte swizzle)
//              into a 4-stage shared-memory ring, completion on mbarriers;
//   warp 1     MMA issuer: one thread issues tcgen05.mma (M=128, N=256,
//              K=16) into a TMEM accumulator, double-buffered (2 x 256
//              columns) so the epilogue of tile i overlaps the mainloop of
//              tile i+1; tcgen05.commit frees smem stages / signals the
//              epilogue;
//   warps 2-5  epilogue: tcgen05.ld of their 32-lane TMEM quarter (one row
//              per thread), fused op, global store.
// Fused epilogues used by the backbone block:
//   EPI_BF16   C -> bf16
//   EPI_F32    C -> fp32
//   EPI_RESID  x[M, N] (fp32 residual stream) += C
//   EPI_GLU    weights interleaved in 128-row gate/up blocks: out[M, N/2] =
//              act(C_gate) * C_up -> bf16   (SwiGLU / tanh-GeGLU)
//   EPI_ROPE   the fused Q|K|V projection: rotate-half RoPE at each row's
//              position on columns < rope_cols, then bf16
// Every output element's K reduction runs in the same order whatever M is
// or where the row sits, so packed (grouped) and per-tenant runs agree
// bit for bit.
#include <mutex>

#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

namespace gemm {
constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 512;  // two 256-column fp32 accumulators
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/;
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);
}  // namespace gemm

// Tile order: groups of `group_m` row-blocks, N fastest inside a group, so
// the CTAs resident at one time share a few A row-blocks and a band of B.
__device__ __forceinline__ void tile_coords(int tile, int num_m, int num_n, int group_m, int& mb,
                                            int& nb) {
    const int per_group = group_m * num_n;
    const int grp = tile / per_group;
    const int first_m = grp * group_m;
    const int gm = min(group_m, num_m - first_m);
    const int in = tile - grp * per_group;
    mb = first_m + in % gm;
    nb = in / gm;
}

__device__ __forceinline__ float act_fn(float g, int act) {
    if (act == JNX_GLU_SWIGLU) return g / (1.0f + expf(-g));
    const float c = 0.7978845608028654f;  // sqrt(2/pi)
    return 0.5f * g * (1.0f + tanhf(c * (g + 0.044715f * g * g * g)));
}

// LoRA up-projection for 32 consecutive columns [col, col + 32) of one row:
// v[e] += t[row, part r..] . B_part[tenant][col + e - part start, :].  The
// 32 columns never straddle two parts (part widths are multiples of 64).
__device__ __forceinline__ void lora_chunk(float (&v)[32], int row, int tenant, int col,
                                           const GemmParams& p) {
    constexpr int R = kLoraRank;
    int part = 0, c = col;
    while (part < 2 && c >= p.lora_cols[part]) {
        c -= p.lora_cols[part];
        ++part;
    }
    const float4* tr = reinterpret_cast<const float4*>(p.lora_t + (size_t)row * p.ldt + part * R);
    float t[R];
#pragma unroll
    for (int i = 0; i < R / 4; ++i) {
        const float4 q = tr[i];
        t[4 * i] = q.x;
        t[4 * i + 1] = q.y;
        t[4 * i + 2] = q.z;
        t[4 * i + 3] = q.w;
    }
    const uint4* b = reinterpret_cast<const uint4*>(
        p.lora_b[part] + ((size_t)tenant * p.lora_cols[part] + c) * R);
#pragma unroll
    for (int e = 0; e < 32; ++e) {
        float acc = 0.f;
#pragma unroll
        for (int h = 0; h < R / 8; ++h) {
            const uint4 w = __ldg(b + (R / 8) * e + h);
            acc += t[8 * h + 0] * __uint_as_float(w.x << 16) +
                   t[8 * h + 1] * __uint_as_float(w.x & 0xFFFF0000u) +
                   t[8 * h + 2] * __uint_as_float(w.y << 16) +
                   t[8 * h + 3] * __uint_as_float(w.y & 0xFFFF0000u) +
                   t[8 * h + 4] * __uint_as_float(w.z << 16) +
                   t[8 * h + 5] * __uint_as_float(w.z & 0xFFFF0000u) +
                   t[8 * h + 6] * __uint_as_float(w.w << 16) +
                   t[8 * h + 7] * __uint_as_float(w.w & 0xFFFF0000u);
        }
        v[e] += acc;
    }
}

template <int EPI, bool LORA>
__device__ __forceinline__ void epilogue_tile(uint32_t tbase, int row, int n0,
                                              const GemmParams& p) {
    const bool valid = row < p.M;
    const int tenant = (LORA && valid) ? p.row_tenant[row] : 0;
    if constexpr (EPI == EPI_BF16 || EPI == EPI_F32 || EPI == EPI_RESID) {
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
            uint32_t r[32];
            tmem_ld32(tbase + c * 32, r);
            tmem_ld_wait();
            if (!valid) continue;
            const int col = n0 + c * 32;
            if constexpr (LORA) {
                float f[32];
#pragma unroll
                for (int e = 0; e < 32; ++e) f[e] = __uint_as_float(r[e]);
                lora_chunk(f, row, tenant, col, p);
#pragma unroll
                for (int e = 0; e < 32; ++e) r[e] = __float_as_uint(f[e]);
            }
            if constexpr (EPI == EPI_BF16) {
                uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16_t*>(p.out) +
                                                      (size_t)row * p.ldo + col);
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    uint4 w;
                    w.x = pack_bf2(__uint_as_float(r[8 * v + 0]), __uint_as_float(r[8 * v + 1]));
                    w.y = pack_bf2(__uint_as_float(r[8 * v + 2]), __uint_as_float(r[8 * v + 3]));
                    w.z = pack_bf2(__uint_as_float(r[8 * v + 4]), __uint_as_float(r[8 * v + 5]));
                    w.w = pack_bf2(__uint_as_float(r[8 * v + 6]), __uint_as_float(r[8 * v + 7]));
                    dst[v] = w;
                }
            } else if constexpr (EPI == EPI_F32) {
                float4* dst = reinterpret_cast<float4*>(static_cast<float*>(p.out) +
                                                        (size_t)row * p.ldo + col);
#pragma unroll
                for (int v = 0; v < 8; ++v)
                    dst[v] = make_float4(__uint_as_float(r[4 * v]), __uint_as_float(r[4 * v + 1]),
                                         __uint_as_float(r[4 * v + 2]),
                                         __uint_as_float(r[4 * v + 3]));
            } else {
                float4* dst = reinterpret_cast<float4*>(p.resid + (size_t)row * p.ldr + col);
#pragma unroll
                for (int v = 0; v < 8; ++v) {
                    float4 x = dst[v];
                    x.x += __uint_as_float(r[4 * v]);
                    x.y += __uint_as_float(r[4 * v + 1]);
                    x.z += __uint_as_float(r[4 * v + 2]);
                    x.w += __uint_as_float(r[4 * v + 3]);
                    dst[v] = x;
                }
            }
        }
    } else if constexpr (EPI == EPI_GLU) {
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            uint32_t g[32], u[32];
            tmem_ld32(tbase + c * 32, g);
            tmem_ld32(tbase + (c + 4) * 32, u);
            tmem_ld_wait();
            if (!valid) continue;
            uint4* dst = reinterpret_cast<uint4*>(static_cast<bf16_t*>(p.out) +
                                                  (size_t)row * p.ldo + n0 / 2 + c * 32);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                float o[8];
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    o[e] = act_fn(__uint_as_float(g[8 * v + e]), p.act) *
                           __uint_as_float(u[8 * v + e]);
                uint4 w;
                w.x = pack_bf2(o[0], o[1]);
                w.y = pack_bf2(o[2], o[3]);
                w.z = pack_bf2(o[4], o[5]);
                w.w = pack_bf2(o[6], o[7]);
                dst[v] = w;
            }
        }
    } else if constexpr (EPI == EPI_ROPE) {
        const int hc = p.hd / 64;  // 32-column chunks in half a head
        const int half = p.hd / 2;
        const int pos = valid ? p.pos[row] : 0;
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
            const int hchunk = c % (2 * hc);
            if (hchunk >= hc) continue;  // handled with its lower partner
            const int col = n0 + c * 32;
            const bool rot = valid && col < p.rope_cols;
            // (cos, sin) of this row's position, 16-byte loads issued before
            // the TMEM read so their latency overlaps it
            float4 cs[16];
            if (rot) {
                const float4* src =
                    reinterpret_cast<const float4*>(p.rope + (size_t)pos * half + hchunk * 32);
#pragma unroll
                for (int e = 0; e < 16; ++e) cs[e] = __ldg(src + e);
            }
            uint32_t lo[32], hi[32];
            tmem_ld32(tbase + c * 32, lo);
            tmem_ld32(tbase + (c + hc) * 32, hi);
            tmem_ld_wait();
            if (!valid) continue;
            float a[32], b[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                a[e] = __uint_as_float(lo[e]);
                b[e] = __uint_as_float(hi[e]);
            }
            if constexpr (LORA) {
                lora_chunk(a, row, tenant, col, p);
                lora_chunk(b, row, tenant, col + half, p);
            }
            if (rot) {
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float cr = (e & 1) ? cs[e >> 1].z : cs[e >> 1].x;
                    const float sr = (e & 1) ? cs[e >> 1].w : cs[e >> 1].y;
                    const float x0 = a[e], x1 = b[e];
                    a[e] = x0 * cr - x1 * sr;
                    b[e] = x1 * cr + x0 * sr;
                }
            }
            bf16_t* base = static_cast<bf16_t*>(p.out) + (size_t)row * p.ldo;
            uint4* d0 = reinterpret_cast<uint4*>(base + col);
            uint4* d1 = reinterpret_cast<uint4*>(base + col + half);
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                uint4 w;
                w.x = pack_bf2(a[8 * v + 0], a[8 * v + 1]);
                w.y = pack_bf2(a[8 * v + 2], a[8 * v + 3]);
                w.z = pack_bf2(a[8 * v + 4], a[8 * v + 5]);
                w.w = pack_bf2(a[8 * v + 6], a[8 * v + 7]);
                d0[v] = w;
                w.x = pack_bf2(b[8 * v + 0], b[8 * v + 1]);
                w.y = pack_bf2(b[8 * v + 2], b[8 * v + 3]);
                w.z = pack_bf2(b[8 * v + 4], b[8 * v + 5]);
                w.w = pack_bf2(b[8 * v + 6], b[8 * v + 7]);
                d1[v] = w;
            }
        }
    }
}

template <int EPI, bool LORA>
__global__ void __launch_bounds__(192, 1)
    k_gemm(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
           GemmParams p) {
    using namespace gemm;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint64_t* full = reinterpret_cast<uint64_t*>(smem + STAGES * STAGE_BYTES);
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* consumed = abort_flag + 1;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 128);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        *consumed = 0;
        fence_barrier_init();
        fence_proxy_async();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, TMEM_COLS);
        tmem_relinquish();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&ta);
        tma_prefetch_desc(&tb);
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    const int num_m = (p.M + BM - 1) / BM;
    const int num_n = p.N / BN;
    const int num_k = p.K / BK;
    const int num_tiles = num_m * num_n;
    int issued = 0;

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            for (int tile = blockIdx.x; tile < num_tiles && !*abort_flag; tile += gridDim.x) {
                int mb, nb;
                tile_coords(tile, num_m, num_n, p.group_m, mb, nb);
                for (int kb = 0; kb < num_k; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1)) {
                        *abort_flag = 1;
                        report(p.status, JNX_ERR_TIMEOUT);
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
                    uint8_t* sa = smem + stage * STAGE_BYTES;
                    tma_load_2d(sa, &ta, kb * BK, mb * BM, &full[stage]);
                    tma_load_2d(sa + A_BYTES, &tb, kb * BK, nb * BN, &full[stage]);
                    ++issued;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int local = 0;
            for (int tile = blockIdx.x; tile < num_tiles && !*abort_flag;
                 tile += gridDim.x, ++local) {
                const int acc = local & 1;
                const uint32_t acc_phase = (local >> 1) & 1;
                if (!mbar_wait(&tempty[acc], acc_phase ^ 1)) {
                    *abort_flag = 1;
                    report(p.status, JNX_ERR_TIMEOUT);
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + acc * BN;
                bool ok = true;
                for (int kb = 0; kb < num_k; ++kb) {
                    if (!mbar_wait(&full[stage], phase)) {
                        ok = false;
                        break;
                    }
                    *consumed = *consumed + 1;
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + stage * STAGE_BYTES);
                    const uint32_t b_addr = a_addr + A_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        tc_mma_f16(d, sw128_desc(a_addr + kk * 32), sw128_desc(b_addr + kk * 32),
                                   IDESC, (kb | kk) != 0);
                    tc_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) {
                    *abort_flag = 1;
                    report(p.status, JNX_ERR_TIMEOUT);
                    break;
                }
                tc_commit(&tfull[acc]);
            }
            // make sure no MMA is still writing TMEM before teardown
            tc_commit(drain);
            mbar_wait(drain, 0);
        }
    } else {
        const int q = warp & 3;  // TMEM lane quarter this warp may access
        int local = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
            const int acc = local & 1;
            const uint32_t acc_phase = (local >> 1) & 1;
            int mb, nb;
            tile_coords(tile, num_m, num_n, p.group_m, mb, nb);
            const int row = mb * BM + q * 32 + lane;
            if (!mbar_wait(&tfull[acc], acc_phase) || *abort_flag) {
                *abort_flag = 1;
                report(p.status, JNX_ERR_TIMEOUT);
                break;
            }
            tc_fence_after();
            epilogue_tile<EPI, LORA>(tmem_base + acc * BN + ((uint32_t)(q * 32) << 16), row,
                                     nb * BN, p);
            tc_fence_before();
            mbar_arrive(&tempty[acc]);
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (*abort_flag && warp == 0 && lane == 0) {
        // wait (bounded) for TMA copies this CTA issued but nobody consumed
        for (int i = *consumed; i < issued; ++i)
            mbar_wait(&full[i % STAGES], (i / STAGES) & 1, 100000000LL);
    }
    __syncwarp();
    if (warp == 1) tmem_dealloc(tmem_base, TMEM_COLS);
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

typedef CUresult (*PFN_tmapEncodeTiled)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                        const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                        const cuuint32_t*, CUtensorMapInterleave,
                                        CUtensorMapSwizzle, CUtensorMapL2promotion,
                                        CUtensorMapFloatOOBfill);

static PFN_tmapEncodeTiled encode_fn() {
    static PFN_tmapEncodeTiled fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        cudaDriverEntryPointQueryResult q;
        void* f = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_tmapEncodeTiled>(f);
    });
    return fn;
}

bool make_tmap_bf16(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols,
                    uint64_t row_stride_elems, uint32_t box_rows, uint32_t box_cols) {
    PFN_tmapEncodeTiled fn = encode_fn();
    if (!fn) return false;
    if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((row_stride_elems * 2) & 15)) return false;
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride_elems * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

template <int EPI, bool LORA = false>
static cudaError_t launch_epi(const CUtensorMap& ta, const CUtensorMap& tb, const GemmParams& p,
                              int grid, cudaStream_t s) {
    static bool attr_done = false;  // per instantiation; idempotent if raced
    if (!attr_done) {
        cudaError_t e = cudaFuncSetAttribute(
            k_gemm<EPI, LORA>, cudaFuncAttributeMaxDynamicSharedMemorySize, gemm::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_done = true;
    }
    k_gemm<EPI, LORA><<<grid, 192, gemm::SMEM_BYTES, s>>>(ta, tb, p);
    return cudaGetLastError();
}

jnx_status gemm_check(int M, int N, int K) {
    if (M < 0 || N <= 0 || K <= 0 || N % gemm::BN || K % gemm::BK)
        return fail(JNX_ERR_UNSUPPORTED, "gemm: need N %% 256 == 0 and K %% 64 == 0 (M=%d N=%d K=%d)",
                    M, N, K);
    return JNX_OK;
}

jnx_status gemm_launch(const uint16_t* A, int lda, const uint16_t* B, int ldb, GemmParams p,
                       cudaStream_t s, int max_ctas) {
    jnx_status st = gemm_check(p.M, p.N, p.K);
    if (st != JNX_OK) return st;
    if (p.M == 0) return JNX_OK;
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, A, p.M, p.K, lda, gemm::BM, gemm::BK) ||
        !make_tmap_bf16(&tb, B, p.N, p.K, ldb, gemm::BN, gemm::BK))
        return fail(JNX_ERR_CUDA, "gemm: tensor map encode failed (alignment or driver)");
    const int tiles = ((p.M + gemm::BM - 1) / gemm::BM) * (p.N / gemm::BN);
    int grid = num_sms();
    if (max_ctas > 0 && max_ctas < grid) grid = max_ctas;
    if (tiles < grid) grid = tiles;
    if (p.group_m <= 0) p.group_m = 16;
    cudaError_t e;
    if (p.lora_t) {
        if (p.epi == EPI_ROPE)
            e = launch_epi<EPI_ROPE, true>(ta, tb, p, grid, s);
        else if (p.epi == EPI_RESID)
            e = launch_epi<EPI_RESID, true>(ta, tb, p, grid, s);
        else
            return fail(JNX_ERR_UNSUPPORTED, "gemm: LoRA only with the RoPE or residual epilogue");
        if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
        return JNX_OK;
    }
    switch (p.epi) {
        case EPI_BF16: e = launch_epi<EPI_BF16>(ta, tb, p, grid, s); break;
        case EPI_F32: e = launch_epi<EPI_F32>(ta, tb, p, grid, s); break;
        case EPI_RESID: e = launch_epi<EPI_RESID>(ta, tb, p, grid, s); break;
        case EPI_GLU: e = launch_epi<EPI_GLU>(ta, tb, p, grid, s); break;
        case EPI_ROPE: e = launch_epi<EPI_ROPE>(ta, tb, p, grid, s); break;
        default: return fail(JNX_ERR_INVALID_ARG, "gemm: unknown epilogue %d", p.epi);
    }
    if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
    return JNX_OK;
}

}  // namespace jnx
