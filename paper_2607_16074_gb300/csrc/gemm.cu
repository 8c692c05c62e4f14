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
// and by the training paths (the GLU's backward, with the gate/up GEMM
// recomputed): EPI_GLU_SAVE (the multipliers u act'(g) | act(g)),
// EPI_GLU_BWD (dm times those multipliers), EPI_GLU_DM (the gate/up
// product times a dm already stored in the up columns).
// Every output element's K reduction runs in the same order whatever M is
// or where the row sits, so packed (grouped) and per-tenant runs agree
// bit for bit.
#include <mutex>
#include <type_traits>

#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

namespace gemm {
constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int TMEM_COLS = 512;  // two 256-column fp32 accumulators
constexpr int STG_BYTES = 4 * 2048;  // epilogue staging, 2 KB per epilogue warp (4 warps)
constexpr int SMEM_BYTES = STAGES * STAGE_BYTES + 1024 /*align*/ + 256 /*barriers*/ + STG_BYTES;
// with eight epilogue warps (two per TMEM lane quarter, each taking half of
// a tile's columns) for the epilogues whose column halves are independent;
// their staging slots are 4 KB (32 rows x 32 fp32 columns)
constexpr int STG_SLOT_EW8 = 4096;
constexpr int SMEM_BYTES_EW8 = SMEM_BYTES - STG_BYTES + 8 * STG_SLOT_EW8;
static_assert(SMEM_BYTES_EW8 <= 227 * 1024, "shared memory per CTA");
constexpr uint32_t IDESC = idesc_bf16_f32(BM, BN);
// LoRA operands of one tile (K = 16, 32-byte rows): t rows and B rows, a
// 2-deep ring after the main stages.
constexpr int LT_BYTES = BM * 16 * 2;
constexpr int LB_BYTES = BN * 16 * 2;
constexpr int LSTAGE = LT_BYTES + LB_BYTES;
constexpr int SMEM_BYTES_LORA = SMEM_BYTES + 2 * LSTAGE;
}  // namespace gemm

// Descriptor of a K-major bf16 tile with 32-byte rows (K = 16) stored with
// the 32-byte swizzle: 8-row atoms of 256 bytes.
__device__ __forceinline__ uint64_t sw32_desc(uint32_t smem_addr) {
    uint64_t d = 0;
    d |= (uint64_t)((smem_addr & 0x3FFFF) >> 4);
    d |= (uint64_t)1 << 16;              // leading byte offset (unused: K fits one row)
    d |= (uint64_t)(256 >> 4) << 32;     // stride byte offset: next 8-row atom
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)6 << 61;              // layout: 32-byte swizzle
    return d;
}

struct NoLora {};

// Rows [row0, row_end) and column block nb of one output tile.  Without
// LoRA, tiles are plain 128-row blocks of M; with LoRA they are laid out per
// tenant segment so every tile belongs to one tenant (`seg`).
struct TileGeo {
    int row0, row_end, nb, seg;
};

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

// Both activations are g sigmoid(z): SiLU with z = g, and the tanh-form
// GELU 0.5 g (1 + tanh(u)) with z = 2 u, u = sqrt(2/pi) (g + 0.044715 g^3),
// since 0.5 (1 + tanh(u)) = sigmoid(2 u).  The sigmoid takes the fast
// exponential and an approximate reciprocal (a few ulp, far below the bf16
// rounding of every product that reads it); its limits are exact (an
// overflowing exponential gives 0).
__device__ __forceinline__ float sigmoid_fast(float z) {
    return __fdividef(1.0f, 1.0f + __expf(-z));
}
__device__ __forceinline__ float gelu_arg(float g) {
    return 1.5957691216057308f * (g + 0.044715f * g * g * g);  // 2 sqrt(2/pi) (g + a g^3)
}

__device__ __forceinline__ float act_fn(float g, int act) {
    return g * sigmoid_fast(act == JNX_GLU_SWIGLU ? g : gelu_arg(g));
}

// act(g) and its derivative, s = sigmoid(z): SiLU' = s (1 + g (1 - s)); for
// the GELU, with tanh(u) = 2 s - 1 and 1 - tanh(u)^2 = 4 s (1 - s),
// d/dg [0.5 g (1 + tanh(u))] = s + 2 g s (1 - s) sqrt(2/pi) (1 + 3 a g^2).
__device__ __forceinline__ void act_grad(float g, int act, float& a, float& da) {
    if (act == JNX_GLU_SWIGLU) {
        const float s = sigmoid_fast(g);
        a = g * s;
        da = s * (1.0f + g * (1.0f - s));
    } else {
        const float s = sigmoid_fast(gelu_arg(g));
        a = g * s;
        da = s + 2.0f * g * s * (1.0f - s) * 0.7978845608028654f *
                     (1.0f + 3.0f * 0.044715f * g * g);
    }
}

// Epilogue staging: each epilogue warp turns its 32 rows x 64 bytes from
// one-row-per-thread (the TMEM layout) into row-contiguous global accesses
// through a 2 KB shared-memory slot.  Writer: thread `lane` puts row `lane`.
// Reader: in step i (0..3) thread `lane` takes row 8 i + lane / 4, 16-byte
// unit lane % 4, so one instruction touches 8 rows x 64 contiguous bytes
// instead of 32 rows x 16 bytes.  Units are XOR-swizzled by (row / 2) % 4,
// which keeps both sides free of bank conflicts.
__device__ __forceinline__ void stg_put(uint8_t* stg, int lane, const uint4 (&v)[4]) {
    uint8_t* rowp = stg + lane * 64;
    const int sw = (lane >> 1) & 3;
#pragma unroll
    for (int j = 0; j < 4; ++j) *reinterpret_cast<uint4*>(rowp + ((j ^ sw) << 4)) = v[j];
}

__device__ __forceinline__ uint4 stg_get(const uint8_t* stg, int lane, int i) {
    const int r = 8 * i + (lane >> 2), j = lane & 3;
    return *reinterpret_cast<const uint4*>(stg + r * 64 + ((j ^ ((r >> 1) & 3)) << 4));
}

__device__ __forceinline__ uint4 pack8_bf16(const float* f) {
    uint4 w;
    w.x = pack_bf2(f[0], f[1]);
    w.y = pack_bf2(f[2], f[3]);
    w.z = pack_bf2(f[4], f[5]);
    w.w = pack_bf2(f[6], f[7]);
    return w;
}

// 32 bf16 per row (64 bytes) from this thread's row to rows row_base + 0..31
// at column `col` of a bf16 [*, ldo] matrix.
__device__ __forceinline__ void stg_store_bf16(uint8_t* stg, int lane, const uint4 (&v)[4],
                                               bf16_t* out, int ldo, int row_base, int row_end,
                                               int col, uint64_t pol) {
    stg_put(stg, lane, v);
    __syncwarp();
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 w = stg_get(stg, lane, i);
        const int row = row_base + 8 * i + (lane >> 2);
        if (row < row_end) st_global_u4_hint(out + (size_t)row * ldo + col + (lane & 3) * 8, w, pol);
    }
    __syncwarp();
}

// RMSNorm factor of a row whose A row is y = bf16(x * gamma) (folded norm):
// rsqrt(mean(x^2) + eps) from the row's partial sums of squares, added in a
// fixed order; 1 without a folded norm.
__device__ __forceinline__ float row_norm_scale(const GemmParams& p, int row, bool valid) {
    if (p.ss_in == nullptr || !valid) return 1.f;
    const float* sp = p.ss_in + (size_t)row * p.ss_parts;
    float t = 0.f;
    for (int i = 0; i < p.ss_parts; ++i) t += sp[i];
    return rsqrtf(t / (float)p.ss_cols + p.ss_eps);
}

// The accumulator tile at tbase (this warp's 32 TMEM lanes = rows
// row_base..row_base+31, 256 fp32 columns) -> the epilogue's output.
// NC, cb: the 32-column chunks [cb, cb + NC) of the tile this warp handles
// (all 8, or one half of 4 with eight epilogue warps: EPI_BF16, EPI_F32,
// EPI_RESID without a folded norm, EPI_GLU_BWD and EPI_GLU_DM only).  Ring slots are
// indexed by the pass within this warp's range, so they stay compile-time.
template <int EPI, int NC = 8>
__device__ __forceinline__ void epilogue_tile(uint32_t tbase, uint8_t* stg, int lane,
                                              int row_base, int row_end, int n0,
                                              const GemmParams& p, int cb = 0) {
    const int my_row = row_base + lane;
    const bool valid = my_row < row_end;
    const uint64_t pol = l2_evict_first_policy();  // outputs and residual are streamed
    if constexpr (EPI == EPI_BF16) {
#pragma unroll 1
        for (int c = cb; c < cb + NC; ++c) {
            uint32_t r[32];
            tmem_ld32(tbase + c * 32, r);
            tmem_ld_wait();
            uint4 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) v[u] = pack8_bf16(reinterpret_cast<const float*>(r) + 8 * u);
            // a 32-column chunk never straddles a 128-column block
            const int n = n0 + c * 32;
            const int col = p.pack_up ? 256 * (n / 128) + 128 + n % 128 : n;
            stg_store_bf16(stg, lane, v, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           col, pol);
        }
    } else if constexpr (EPI == EPI_F32 || EPI == EPI_RESID) {
        // 16 fp32 columns (64 bytes) per staging pass; the residual is
        // loaded RD - 1 passes ahead of its use, so several passes' loads
        // are in flight while the accumulator is staged (a shallower ring for
        // half-tile warps, which run with fewer registers per thread)
        constexpr int RD = NC == 4 ? 3 : 4;
        float* dst = EPI == EPI_RESID ? p.resid : static_cast<float*>(p.out);
        const int ld = EPI == EPI_RESID ? p.ldr : p.ldo;
        float4 xr[RD][4];
        uint2 gr[RD];  // folded norm: this lane's four gamma values of each pass
        const bool norm = EPI == EPI_RESID && p.norm_gamma != nullptr;
        auto load_resid = [&](int pass, float4 (&x)[4], uint2& gq) {
            const int col = n0 + pass * 16 + (lane & 3) * 4;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int row = row_base + 8 * i + (lane >> 2);
                uint4 u = make_uint4(0u, 0u, 0u, 0u);
                if (row < row_end) u = ld_global_u4_hint(dst + (size_t)row * ld + col, pol);
                x[i] = make_float4(__uint_as_float(u.x), __uint_as_float(u.y),
                                   __uint_as_float(u.z), __uint_as_float(u.w));
            }
            if (norm) gq = *reinterpret_cast<const uint2*>(p.norm_gamma + col);
        };
        constexpr int NP = 2 * NC;  // staging passes of this warp
        const int pb = 2 * cb;
        if constexpr (EPI == EPI_RESID) {
#pragma unroll
            for (int q = 0; q < RD - 1; ++q) load_resid(pb + q, xr[q], gr[q]);
        }
        // folded RMSNorm (EPI_RESID with norm_gamma): y = bf16(x * gamma) and
        // the sums of x^2 of each of this lane's four rows over its columns,
        // one per 128-column half of the tile (8 staging passes each)
        float ssq[NC / 4][4] = {};
#pragma unroll
        for (int lc = 0; lc < NC; ++lc) {
            const int c = cb + lc;
            uint32_t r[32];
            tmem_ld32(tbase + c * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int lp = 2 * lc + h;  // pass within this warp's range
                const int pass = pb + lp;
                if constexpr (EPI == EPI_RESID)
                    if (lp + RD - 1 < NP)
                        load_resid(pass + RD - 1, xr[(lp + RD - 1) % RD], gr[(lp + RD - 1) % RD]);
                uint4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    v[u] = make_uint4(r[16 * h + 4 * u], r[16 * h + 4 * u + 1],
                                      r[16 * h + 4 * u + 2], r[16 * h + 4 * u + 3]);
                stg_put(stg, lane, v);
                __syncwarp();
                const int col = n0 + pass * 16 + (lane & 3) * 4;
                float gf[4] = {0.f, 0.f, 0.f, 0.f};
                if (EPI == EPI_RESID && norm) {
                    const uint2 g = gr[lp % RD];
                    gf[0] = bf2f(g.x & 0xFFFF);
                    gf[1] = bf2f(g.x >> 16);
                    gf[2] = bf2f(g.y & 0xFFFF);
                    gf[3] = bf2f(g.y >> 16);
                }
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 w = stg_get(stg, lane, i);
                    const int row = row_base + 8 * i + (lane >> 2);
                    float4 o = make_float4(__uint_as_float(w.x), __uint_as_float(w.y),
                                           __uint_as_float(w.z), __uint_as_float(w.w));
                    if constexpr (EPI == EPI_RESID) {
                        const float4 x = xr[lp % RD][i];
                        o.x += x.x;
                        o.y += x.y;
                        o.z += x.z;
                        o.w += x.w;
                    }
                    if (row < row_end)
                        st_global_u4_hint(dst + (size_t)row * ld + col,
                                          make_uint4(__float_as_uint(o.x), __float_as_uint(o.y),
                                                     __float_as_uint(o.z), __float_as_uint(o.w)),
                                          pol);
                    if (EPI == EPI_RESID && norm) {
                        ssq[lp / 8][i] += o.x * o.x + o.y * o.y + o.z * o.z + o.w * o.w;
                        if (row < row_end)
                            *reinterpret_cast<uint2*>(p.norm_out + (size_t)row * p.N + col) =
                                make_uint2(pack_bf2(o.x * gf[0], o.y * gf[1]),
                                           pack_bf2(o.z * gf[2], o.w * gf[3]));
                    }
                }
                __syncwarp();
            }
        }
        if (norm) {
            // the four lanes of a row hold each half's columns between them
            const int parts = p.N / 128;
#pragma unroll
            for (int hb = 0; hb < NC / 4; ++hb)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    float t = ssq[hb][i];
                    t += __shfl_xor_sync(0xffffffffu, t, 1);
                    t += __shfl_xor_sync(0xffffffffu, t, 2);
                    const int row = row_base + 8 * i + (lane >> 2);
                    if ((lane & 3) == 0 && row < row_end)
                        p.ss_out[(size_t)row * parts + (n0 + 32 * cb) / 128 + hb] = t;
                }
        }
    } else if constexpr (EPI == EPI_GLU) {
        const float rs = row_norm_scale(p, my_row, valid);
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            uint32_t g[32], u[32];
            tmem_ld32(tbase + c * 32, g);
            tmem_ld32(tbase + (c + 4) * 32, u);
            tmem_ld_wait();
            uint4 v[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float o[8];
#pragma unroll
                for (int e = 0; e < 8; ++e)
                    o[e] = act_fn(rs * __uint_as_float(g[8 * q + e]), p.act) *
                           (rs * __uint_as_float(u[8 * q + e]));
                v[q] = pack8_bf16(o);
            }
            stg_store_bf16(stg, lane, v, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           n0 / 2 + c * 32, pol);
        }
    } else if constexpr (EPI == EPI_GLU_SAVE) {
        const float rs = row_norm_scale(p, my_row, valid);
#pragma unroll 1
        for (int c = 0; c < 4; ++c) {
            uint32_t g[32], u[32];
            tmem_ld32(tbase + c * 32, g);
            tmem_ld32(tbase + (c + 4) * 32, u);
            tmem_ld_wait();
            uint4 vg[4], vu[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                float og[8], ou[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float a, da;
                    act_grad(rs * __uint_as_float(g[8 * q + e]), p.act, a, da);
                    og[e] = rs * __uint_as_float(u[8 * q + e]) * da;
                    ou[e] = a;
                }
                vg[q] = pack8_bf16(og);
                vu[q] = pack8_bf16(ou);
            }
            stg_store_bf16(stg, lane, vg, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           n0 + c * 32, pol);
            stg_store_bf16(stg, lane, vu, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           n0 + 128 + c * 32, pol);
        }
    } else if constexpr (EPI == EPI_GLU_DM) {
        // as EPI_GLU_SAVE over the chunk pairs (gate c, up c + 4) of this
        // warp's range (all four, or two of them with eight epilogue warps),
        // with dm (this thread's row, the chunk's 32 F columns: 64
        // contiguous bytes of the up slot, through L1 so each 32-byte sector
        // is fetched once) loaded one chunk ahead; every lane of the warp has
        // its chunk's dm in registers before any lane's stores reach that
        // chunk's columns, so out may be aux
        const int c0 = cb / 2, nc = NC / 2;
        const float rs = row_norm_scale(p, my_row, valid);
        const bf16_t* dmrow = p.aux + (size_t)my_row * p.ldaux + n0 + 128;
        uint4 dmv[2][4];
        auto load_dm = [&](int c, uint4 (&v)[4]) {
#pragma unroll
            for (int q = 0; q < 4; ++q)
                v[q] = valid ? *reinterpret_cast<const uint4*>(dmrow + c * 32 + 8 * q)
                             : make_uint4(0u, 0u, 0u, 0u);
        };
        load_dm(c0, dmv[0]);
#pragma unroll
        for (int lc = 0; lc < nc; ++lc) {
            const int c = c0 + lc;
            uint32_t g[32], u[32];
            tmem_ld32(tbase + c * 32, g);
            tmem_ld32(tbase + (c + 4) * 32, u);
            if (lc + 1 < nc) load_dm(c + 1, dmv[(lc + 1) & 1]);
            tmem_ld_wait();
            uint4 vg[4], vu[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const uint4 m4 = dmv[lc & 1][q];
                const uint32_t mw[4] = {m4.x, m4.y, m4.z, m4.w};
                float og[8], ou[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    float a, da;
                    act_grad(rs * __uint_as_float(g[8 * q + e]), p.act, a, da);
                    const float dm = bf2f((mw[e / 2] >> (16 * (e & 1))) & 0xFFFF);
                    og[e] = dm * (rs * __uint_as_float(u[8 * q + e]) * da);
                    ou[e] = dm * a;
                }
                vg[q] = pack8_bf16(og);
                vu[q] = pack8_bf16(ou);
            }
            stg_store_bf16(stg, lane, vg, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           n0 + c * 32, pol);
            stg_store_bf16(stg, lane, vu, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           n0 + 128 + c * 32, pol);
        }
    } else if constexpr (EPI == EPI_GLU_BWD && NC == 4) {
        // half-tile warps (4 KB staging slot): one staging round per 32-column
        // chunk, so each lane takes 8 contiguous columns of rows 8 i + lane / 4
        // and its multiplier loads and result stores are 16 bytes; the next
        // chunk's multipliers are in flight while one is finished.  F column f
        // has its gate slot at packed column 256 (f / 128) + f % 128, its up
        // slot 128 later; a lane reads each element before it writes it, so
        // out may be aux.
        auto pcol = [&](int c) {
            const int f = n0 + c * 32 + (lane & 3) * 8;
            return (f / 128) * 256 + (f % 128);
        };
        uint4 mg[2][4], mu[2][4];
        auto load_m = [&](int c, uint4 (&g)[4], uint4 (&u)[4]) {
            const int pc = pcol(c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int row = row_base + 8 * i + (lane >> 2);
                g[i] = u[i] = make_uint4(0u, 0u, 0u, 0u);
                if (row < row_end) {
                    const bf16_t* src = p.aux + (size_t)row * p.ldaux + pc;
                    g[i] = ld_global_u4_hint(src, pol);
                    u[i] = ld_global_u4_hint(src + 128, pol);
                }
            }
        };
        load_m(cb, mg[0], mu[0]);
#pragma unroll
        for (int lc = 0; lc < NC; ++lc) {
            const int c = cb + lc;
            if (lc + 1 < NC) load_m(c + 1, mg[(lc + 1) & 1], mu[(lc + 1) & 1]);
            uint32_t r[32];
            tmem_ld32(tbase + c * 32, r);
            tmem_ld_wait();
            // row `lane` puts its 32 fp32 (8 units of 16 bytes, XOR-swizzled
            // by row % 8)
            uint8_t* rowp = stg + lane * 128;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                *reinterpret_cast<uint4*>(rowp + ((j ^ (lane & 7)) << 4)) =
                    make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
            __syncwarp();
            const int pc = pcol(c);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int rr = 8 * i + (lane >> 2), u0 = (lane & 3) * 2;
                const uint8_t* rp = stg + rr * 128;
                const uint4 a = *reinterpret_cast<const uint4*>(rp + ((u0 ^ (rr & 7)) << 4));
                const uint4 b = *reinterpret_cast<const uint4*>(rp + (((u0 + 1) ^ (rr & 7)) << 4));
                const float dm[8] = {__uint_as_float(a.x), __uint_as_float(a.y),
                                     __uint_as_float(a.z), __uint_as_float(a.w),
                                     __uint_as_float(b.x), __uint_as_float(b.y),
                                     __uint_as_float(b.z), __uint_as_float(b.w)};
                const uint4 gm = mg[lc & 1][i], um = mu[lc & 1][i];
                const uint32_t gw[4] = {gm.x, gm.y, gm.z, gm.w};
                const uint32_t uw[4] = {um.x, um.y, um.z, um.w};
                float og[8], ou[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    og[e] = dm[e] * bf2f((gw[e / 2] >> (16 * (e & 1))) & 0xFFFF);
                    ou[e] = dm[e] * bf2f((uw[e / 2] >> (16 * (e & 1))) & 0xFFFF);
                }
                const int row = row_base + rr;
                if (row < row_end) {
                    bf16_t* dst = static_cast<bf16_t*>(p.out) + (size_t)row * p.ldo + pc;
                    st_global_u4_hint(dst, pack8_bf16(og), pol);
                    st_global_u4_hint(dst + 128, pack8_bf16(ou), pol);
                }
            }
            __syncwarp();
        }
    } else if constexpr (EPI == EPI_GLU_BWD) {
        // accumulator: dm for F columns [n0, n0 + 256); F column f has its
        // gate slot at packed column 256 (f / 128) + f % 128 and its up slot
        // 128 later.  As EPI_RESID: 16 columns per pass, dm staged through
        // shared memory so lane handles 4 columns of rows 8 i + lane / 4 (its
        // loads and stores cover 8 rows x 32 contiguous bytes per
        // instruction), the multipliers of pass + RD - 1 in flight.  Each
        // element is read before the same lane writes it, so out may be aux.
        constexpr int RD = 4;
        auto pcol = [&](int pass) {
            const int f = n0 + pass * 16 + (lane & 3) * 4;
            return (f / 128) * 256 + (f % 128);
        };
        uint2 mg[RD][4], mu[RD][4];
        auto load_m = [&](int pass, uint2 (&g)[4], uint2 (&u)[4]) {
            const int pc = pcol(pass);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int row = row_base + 8 * i + (lane >> 2);
                g[i] = u[i] = make_uint2(0u, 0u);
                if (row < row_end) {
                    const bf16_t* src = p.aux + (size_t)row * p.ldaux + pc;
                    g[i] = ld_global_u2_hint(src, pol);
                    u[i] = ld_global_u2_hint(src + 128, pol);
                }
            }
        };
        constexpr int NP = 2 * NC;  // staging passes of this warp
        const int pb = 2 * cb;
#pragma unroll
        for (int q = 0; q < RD - 1; ++q) load_m(pb + q, mg[q], mu[q]);
#pragma unroll
        for (int lc = 0; lc < NC; ++lc) {
            const int c = cb + lc;
            uint32_t r[32];
            tmem_ld32(tbase + c * 32, r);
            tmem_ld_wait();
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int lp = 2 * lc + h;  // pass within this warp's range
                const int pass = pb + lp;
                if (lp + RD - 1 < NP) load_m(pass + RD - 1, mg[(lp + RD - 1) % RD],
                                             mu[(lp + RD - 1) % RD]);
                uint4 v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    v[u] = make_uint4(r[16 * h + 4 * u], r[16 * h + 4 * u + 1],
                                      r[16 * h + 4 * u + 2], r[16 * h + 4 * u + 3]);
                stg_put(stg, lane, v);
                __syncwarp();
                const int pc = pcol(pass);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const uint4 wv = stg_get(stg, lane, i);
                    const int row = row_base + 8 * i + (lane >> 2);
                    const float dm[4] = {__uint_as_float(wv.x), __uint_as_float(wv.y),
                                         __uint_as_float(wv.z), __uint_as_float(wv.w)};
                    const uint2 gm = mg[lp % RD][i], um = mu[lp % RD][i];
                    const uint2 og = make_uint2(
                        pack_bf2(dm[0] * bf2f(gm.x & 0xFFFF), dm[1] * bf2f(gm.x >> 16)),
                        pack_bf2(dm[2] * bf2f(gm.y & 0xFFFF), dm[3] * bf2f(gm.y >> 16)));
                    const uint2 ou = make_uint2(
                        pack_bf2(dm[0] * bf2f(um.x & 0xFFFF), dm[1] * bf2f(um.x >> 16)),
                        pack_bf2(dm[2] * bf2f(um.y & 0xFFFF), dm[3] * bf2f(um.y >> 16)));
                    if (row < row_end) {
                        bf16_t* dst = static_cast<bf16_t*>(p.out) + (size_t)row * p.ldo + pc;
                        st_global_u2_hint(dst, og, pol);
                        st_global_u2_hint(dst + 128, ou, pol);
                    }
                }
                __syncwarp();
            }
        }
    } else if constexpr (EPI == EPI_ROPE) {
        const int hc = p.hd / 64;  // 32-column chunks in half a head
        const int half = p.hd / 2;
        // a position outside the (cos, sin) table is reported and its row
        // is left unrotated (the table load is skipped)
        int pos = valid ? p.pos[my_row] : 0;
        const bool pos_ok = pos >= 0 && pos < p.rope_ld;
        if (valid && !pos_ok) report(p.status, JNX_ERR_DEVICE_BOUNDS);
        if (!pos_ok) pos = 0;
        const float rs = row_norm_scale(p, my_row, valid);
#pragma unroll 1
        for (int c = 0; c < 8; ++c) {
            const int hchunk = c % (2 * hc);
            if (hchunk >= hc) continue;  // handled with its lower partner
            const int col = n0 + c * 32;
            const bool rot = valid && pos_ok && col < p.rope_cols;
            // (cos, sin) of this row's position for the chunk's 32
            // frequencies, loaded before the TMEM read so their latency
            // overlaps it; the table is frequency-major, so the warp's rows
            // (mostly consecutive positions) read consecutive entries
            float2 cs[32];
            if (rot) {
                const float2* src = p.rope + (size_t)(hchunk * 32) * p.rope_ld + pos;
#pragma unroll
                for (int e = 0; e < 32; ++e) cs[e] = __ldg(src + (size_t)e * p.rope_ld);
            }
            uint32_t lo[32], hi[32];
            tmem_ld32(tbase + c * 32, lo);
            tmem_ld32(tbase + (c + hc) * 32, hi);
            tmem_ld_wait();
            float a[32], b[32];
#pragma unroll
            for (int e = 0; e < 32; ++e) {
                a[e] = rs * __uint_as_float(lo[e]);
                b[e] = rs * __uint_as_float(hi[e]);
            }
            if (rot) {
#pragma unroll
                for (int e = 0; e < 32; ++e) {
                    const float cr = cs[e].x, sr = cs[e].y;
                    const float x0 = a[e], x1 = b[e];
                    a[e] = x0 * cr - x1 * sr;
                    b[e] = x1 * cr + x0 * sr;
                }
            }
            uint4 v[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) v[q] = pack8_bf16(a + 8 * q);
            stg_store_bf16(stg, lane, v, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           col, pol);
#pragma unroll
            for (int q = 0; q < 4; ++q) v[q] = pack8_bf16(b + 8 * q);
            stg_store_bf16(stg, lane, v, static_cast<bf16_t*>(p.out), p.ldo, row_base, row_end,
                           col + half, pol);
        }
    }
}

template <bool LORA, class LG>
__device__ __forceinline__ TileGeo tile_geo(int tile, int num_m, int num_n, const GemmParams& p,
                                            const LG& lg) {
    int mb, nb;
    tile_coords(tile, num_m, num_n, p.group_m, mb, nb);
    TileGeo g;
    g.nb = nb;
    if constexpr (LORA) {
        int sg = 0;
        while (sg + 1 < lg.n_seg && lg.seg_tile0[sg + 1] <= mb) ++sg;
        g.seg = sg;
        g.row0 = lg.seg_r0[sg] + (mb - lg.seg_tile0[sg]) * gemm::BM;
        g.row_end = min(g.row0 + gemm::BM, lg.seg_r1[sg]);
    } else {
        g.seg = 0;
        g.row0 = mb * gemm::BM;
        g.row_end = min(g.row0 + gemm::BM, p.M);
    }
    return g;
}

// The LoRA part holding column block nb, and the block's first column in it.
__device__ __forceinline__ void lora_part(const LoraGemm& lg, int nb, int& part, int& c0) {
    int c = nb * gemm::BN;
    part = 0;
    while (part + 1 < lg.n_parts && c >= lg.part_cols[part]) {
        c -= lg.part_cols[part];
        ++part;
    }
    c0 = c;
}

template <int EPI, bool LORA, int EW>
__global__ void __launch_bounds__(64 + 32 * EW, 1)
    k_gemm(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
           const __grid_constant__ typename std::conditional<LORA, LoraGemm, NoLora>::type lg,
           GemmParams p) {
    using namespace gemm;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* lsm = smem + STAGES * STAGE_BYTES;  // LoRA ring (LORA only)
    uint64_t* full = reinterpret_cast<uint64_t*>(lsm + (LORA ? 2 * LSTAGE : 0));
    uint64_t* empty = full + STAGES;
    uint64_t* tfull = empty + STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint64_t* lfull = drain + 1;   // [2]
    uint64_t* lempty = lfull + 2;  // [2]
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(lempty + 2);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    volatile int* consumed = abort_flag + 1;
    volatile int* lconsumed = abort_flag + 2;

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 32 * EW);
            mbar_init(&lfull[a], 1);
            mbar_init(&lempty[a], 1);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        *consumed = 0;
        *lconsumed = 0;
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

    int num_m;
    if constexpr (LORA)
        num_m = lg.seg_tile0[lg.n_seg];
    else
        num_m = (p.M + BM - 1) / BM;
    const int num_n = p.N / BN;
    const int num_k = p.K / BK;
    const int num_tiles = num_m * num_n;
    int issued = 0, l_issued = 0;

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int lj = 0;
            uint32_t lphase = 0;
            for (int tile = blockIdx.x; tile < num_tiles && !*abort_flag; tile += gridDim.x) {
                const TileGeo g = tile_geo<LORA>(tile, num_m, num_n, p, lg);
                for (int kb = 0; kb < num_k; ++kb) {
                    if (!mbar_wait(&empty[stage], phase ^ 1)) {
                        *abort_flag = 1;
                        report(p.status, JNX_ERR_TIMEOUT);
                        break;
                    }
                    mbar_arrive_expect_tx(&full[stage], STAGE_BYTES);
                    uint8_t* sa = smem + stage * STAGE_BYTES;
                    tma_load_2d(sa, &ta, kb * BK, g.row0, &full[stage]);
                    int brow = g.nb * BN;
                    if constexpr (LORA)
                        if (lg.seg_b) brow += lg.seg_tenant[g.seg] * p.N;
                    tma_load_2d(sa + A_BYTES, &tb, kb * BK, brow, &full[stage]);
                    ++issued;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if constexpr (LORA) {
                    if (*abort_flag) break;
                    if (lg.n_parts == 0) continue;  // segmented weights only
                    // this tile's t rows (its part) and its tenant's B rows
                    if (!mbar_wait(&lempty[lj], lphase ^ 1)) {
                        *abort_flag = 1;
                        report(p.status, JNX_ERR_TIMEOUT);
                        break;
                    }
                    int part, c0;
                    lora_part(lg, g.nb, part, c0);
                    uint8_t* lt = lsm + lj * LSTAGE;
                    mbar_arrive_expect_tx(&lfull[lj], LSTAGE);
                    tma_load_2d(lt, &lg.tt, part * 16, g.row0, &lfull[lj]);
                    tma_load_2d(lt + LT_BYTES, &lg.tb[part], 0,
                                lg.seg_tenant[g.seg] * lg.part_cols[part] + c0, &lfull[lj]);
                    ++l_issued;
                    if (++lj == 2) {
                        lj = 0;
                        lphase ^= 1;
                    }
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int local = 0;
            int lj = 0;
            uint32_t lphase = 0;
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
                if constexpr (LORA) {
                    // D += t[rows, part] . B_part[tenant][cols]^T (one K = 16 step);
                    // none with segmented weights only (n_parts == 0)
                    if (ok && lg.n_parts > 0) {
                        if (!mbar_wait(&lfull[lj], lphase)) {
                            ok = false;
                        } else {
                            *lconsumed = *lconsumed + 1;
                            tc_fence_after();
                            const uint32_t la = smem_u32(lsm + lj * LSTAGE);
                            tc_mma_f16(d, sw32_desc(la), sw32_desc(la + LT_BYTES), IDESC, 1);
                            tc_commit(&lempty[lj]);
                            if (++lj == 2) {
                                lj = 0;
                                lphase ^= 1;
                            }
                        }
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
        // with eight epilogue warps, warps 2-5 take chunks 0-3 of a tile and
        // warps 6-9 chunks 4-7 (the same lane quarters)
        const int cb = EW == 8 ? ((warp - 2) >> 2) * 4 : 0;
        // this warp's staging slot, after the barrier block
        uint8_t* stg = reinterpret_cast<uint8_t*>(full) + 256 +
                       (warp - 2) * (EW == 8 ? gemm::STG_SLOT_EW8 : 2048);
        int local = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
            const int acc = local & 1;
            const uint32_t acc_phase = (local >> 1) & 1;
            const TileGeo g = tile_geo<LORA>(tile, num_m, num_n, p, lg);
            const int row_base = g.row0 + q * 32;
            if constexpr (EPI == EPI_GLU_DM) {
                // this thread's dm for the tile (its row, its chunks of the
                // up slot) into L2 while the tile's K loop runs
                const int row = row_base + lane;
                const int nbytes = (EW == 8 ? 2 : 4) * 64;
                if (row < g.row_end)
                    for (int b = 0; b < nbytes; b += 128)
                        prefetch_l2(reinterpret_cast<const uint8_t*>(
                                        p.aux + (size_t)row * p.ldaux + g.nb * BN + 128 + cb * 16) +
                                    b);
            }
            if (!mbar_wait(&tfull[acc], acc_phase) || *abort_flag) {
                *abort_flag = 1;
                report(p.status, JNX_ERR_TIMEOUT);
                break;
            }
            tc_fence_after();
            epilogue_tile<EPI, EW == 8 ? 4 : 8>(tmem_base + acc * BN + ((uint32_t)(q * 32) << 16),
                                                stg, lane, row_base, g.row_end, g.nb * BN, p, cb);
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
        for (int i = *lconsumed; i < l_issued; ++i)
            mbar_wait(&lfull[i & 1], (i >> 1) & 1, 100000000LL);
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
                    uint64_t row_stride_elems, uint32_t box_rows, uint32_t box_cols,
                    int swizzle_bytes) {
    PFN_tmapEncodeTiled fn = encode_fn();
    if (!fn) return false;
    if ((reinterpret_cast<uintptr_t>(ptr) & 15) || ((row_stride_elems * 2) & 15)) return false;
    if (box_cols * 2 > (uint32_t)swizzle_bytes) return false;  // a box row within one swizzle span
    cuuint64_t dims[2] = {cols, rows};
    cuuint64_t strides[1] = {row_stride_elems * 2};
    cuuint32_t box[2] = {box_cols, box_rows};
    cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                  : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                        : CU_TENSOR_MAP_SWIZZLE_32B;
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box,
              estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int num_sms() {
    int dev = 0, n = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    return n > 0 ? n : 1;
}

cudaError_t set_smem_limit(const void* fn, int bytes, std::atomic<uint64_t>& done) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = dev < 64 ? 1ull << dev : 0ull;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) done.fetch_or(bit, std::memory_order_acq_rel);
    return e;
}

template <int EPI, bool LORA, class LG, int EW = 4>
static cudaError_t launch_epi(const CUtensorMap& ta, const CUtensorMap& tb, const LG& lg,
                              const GemmParams& p, int grid, cudaStream_t s) {
    static_assert(EW == 4 || (EW == 8 && !LORA &&
                              (EPI == EPI_BF16 || EPI == EPI_F32 || EPI == EPI_RESID ||
                               EPI == EPI_GLU_BWD || EPI == EPI_GLU_DM)),
                  "eight epilogue warps: column-splittable epilogues without LoRA only");
    constexpr int smem = LORA ? gemm::SMEM_BYTES_LORA
                              : (EW == 8 ? gemm::SMEM_BYTES_EW8 : gemm::SMEM_BYTES);
    static std::atomic<uint64_t> attr{0};  // per instantiation, one bit per device
    cudaError_t e = set_smem_limit(reinterpret_cast<const void*>(k_gemm<EPI, LORA, EW>), smem, attr);
    if (e != cudaSuccess) return e;
    k_gemm<EPI, LORA, EW><<<grid, 64 + 32 * EW, smem, s>>>(ta, tb, lg, p);
    return cudaGetLastError();
}

// Tile-order group height: enough 128-row blocks of A to hold ~40 MB in L2
// while the group sweeps all column blocks, so each weight band is re-read
// once per group rather than once per few row blocks.  Measured on GB300 at
// 65,536 tokens: gate/up (K=4096) 1810 -> ~1870 TFLOP/s going from 16 to 40,
// QKV best at 32-48, down (K=11008) best at 14-16.
static int default_group_m(int K) {
    const double a_block = (double)gemm::BM * K * 2.0;
    int g = (int)(40.0 * 1024 * 1024 / a_block + 0.5);
    return g < 8 ? 8 : (g > 48 ? 48 : g);
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
    if (p.group_m <= 0) p.group_m = default_group_m(p.K);
    cudaError_t e;
    const NoLora none{};
    switch (p.epi) {
        case EPI_BF16: e = launch_epi<EPI_BF16, false>(ta, tb, none, p, grid, s); break;
        // eight epilogue warps only where the epilogue is the bottleneck: with
        // the fp32 and residual epilogues they slowed the GEMMs on GB300 (the
        // 7B-class O / down projections 1,314 / 1,460 -> 1,246 / 1,419 TFLOP/s)
        case EPI_F32: e = launch_epi<EPI_F32, false>(ta, tb, none, p, grid, s); break;
        case EPI_RESID: e = launch_epi<EPI_RESID, false>(ta, tb, none, p, grid, s); break;
        case EPI_GLU: e = launch_epi<EPI_GLU, false>(ta, tb, none, p, grid, s); break;
        case EPI_ROPE: e = launch_epi<EPI_ROPE, false>(ta, tb, none, p, grid, s); break;
        case EPI_GLU_BWD:
            e = launch_epi<EPI_GLU_BWD, false, NoLora, 8>(ta, tb, none, p, grid, s);
            break;
        case EPI_GLU_SAVE: e = launch_epi<EPI_GLU_SAVE, false>(ta, tb, none, p, grid, s); break;
        case EPI_GLU_DM:
            e = launch_epi<EPI_GLU_DM, false, NoLora, 8>(ta, tb, none, p, grid, s);
            break;
        default: return fail(JNX_ERR_INVALID_ARG, "gemm: unknown epilogue %d", p.epi);
    }
    if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
    return JNX_OK;
}

jnx_status gemm_launch_seg(const uint16_t* A, int lda, const uint16_t* B, int ldb, int n_tenants,
                           GemmParams p, int n_seg, const int* seg_r0, const int* seg_r1,
                           const int* seg_tenant, cudaStream_t s) {
    jnx_status st = gemm_check(p.M, p.N, p.K);
    if (st != JNX_OK) return st;
    if (n_seg < 0 || n_seg > kLoraMaxSlots || n_tenants <= 0)
        return fail(JNX_ERR_UNSUPPORTED, "gemm: bad segment description");
    if (p.M == 0 || n_seg == 0) return JNX_OK;
    static thread_local LoraGemm lg;  // staging of the kernel argument (copied at launch)
    lg = LoraGemm{};
    lg.n_parts = 0;
    lg.seg_b = 1;
    lg.n_seg = n_seg;
    int tiles = 0;
    for (int i = 0; i < n_seg; ++i) {
        if (seg_r0[i] < 0 || seg_r1[i] < seg_r0[i] || seg_r1[i] > p.M || seg_tenant[i] < 0 ||
            seg_tenant[i] >= n_tenants)
            return fail(JNX_ERR_INVALID_ARG, "gemm: bad segment %d", i);
        lg.seg_r0[i] = seg_r0[i];
        lg.seg_r1[i] = seg_r1[i];
        lg.seg_tenant[i] = seg_tenant[i];
        lg.seg_tile0[i] = tiles;
        tiles += (seg_r1[i] - seg_r0[i] + gemm::BM - 1) / gemm::BM;
    }
    lg.seg_tile0[n_seg] = tiles;
    CUtensorMap ta, tb;
    if (!make_tmap_bf16(&ta, A, p.M, p.K, lda, gemm::BM, gemm::BK) ||
        !make_tmap_bf16(&tb, B, (uint64_t)n_tenants * p.N, p.K, ldb, gemm::BN, gemm::BK))
        return fail(JNX_ERR_CUDA, "gemm: tensor map encode failed (alignment or driver)");
    const int total = tiles * (p.N / gemm::BN);
    if (total == 0) return JNX_OK;
    int grid = num_sms();
    if (total < grid) grid = total;
    if (p.group_m <= 0) p.group_m = default_group_m(p.K);
    cudaError_t e;
    switch (p.epi) {
        case EPI_BF16: e = launch_epi<EPI_BF16, true>(ta, tb, lg, p, grid, s); break;
        case EPI_F32: e = launch_epi<EPI_F32, true>(ta, tb, lg, p, grid, s); break;
        case EPI_RESID: e = launch_epi<EPI_RESID, true>(ta, tb, lg, p, grid, s); break;
        case EPI_GLU: e = launch_epi<EPI_GLU, true>(ta, tb, lg, p, grid, s); break;
        case EPI_GLU_SAVE: e = launch_epi<EPI_GLU_SAVE, true>(ta, tb, lg, p, grid, s); break;
        case EPI_GLU_BWD: e = launch_epi<EPI_GLU_BWD, true>(ta, tb, lg, p, grid, s); break;
        default: return fail(JNX_ERR_INVALID_ARG, "gemm: epilogue %d unsupported here", p.epi);
    }
    if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
    return JNX_OK;
}

jnx_status gemm_launch_lora(const uint16_t* A, int lda, const uint16_t* B, int ldb, GemmParams p,
                            const LoraSpec& ls, cudaStream_t s) {
    jnx_status st = gemm_check(p.M, p.N, p.K);
    if (st != JNX_OK) return st;
    if (p.epi != EPI_ROPE && p.epi != EPI_RESID)
        return fail(JNX_ERR_UNSUPPORTED, "gemm: LoRA only with the RoPE or residual epilogue");
    if (ls.n_seg < 0 || ls.n_seg > kLoraMaxSlots || ls.n_parts < 1 || ls.n_parts > 3 ||
        (ls.ldt * 2) % 16 || ls.ldt < 16 * ls.n_parts)
        return fail(JNX_ERR_UNSUPPORTED, "gemm: bad LoRA description");
    int cols = 0;
    for (int i = 0; i < ls.n_parts; ++i) {
        if (ls.cols[i] <= 0 || ls.cols[i] % gemm::BN)
            return fail(JNX_ERR_UNSUPPORTED, "gemm: LoRA part widths must be multiples of 256");
        cols += ls.cols[i];
    }
    if (cols != p.N) return fail(JNX_ERR_INVALID_ARG, "gemm: LoRA parts do not cover N");
    if (p.M == 0 || ls.n_seg == 0) return JNX_OK;
    static thread_local LoraGemm lg;  // staging of the kernel argument (copied at launch)
    lg = LoraGemm{};
    lg.n_parts = ls.n_parts;
    lg.n_seg = ls.n_seg;
    int tiles = 0;
    for (int i = 0; i < ls.n_seg; ++i) {
        if (ls.seg_r0[i] < 0 || ls.seg_r1[i] < ls.seg_r0[i] || ls.seg_r1[i] > p.M ||
            ls.seg_tenant[i] < 0 || ls.seg_tenant[i] >= ls.n_tenants)
            return fail(JNX_ERR_INVALID_ARG, "gemm: bad LoRA segment %d", i);
        lg.seg_r0[i] = ls.seg_r0[i];
        lg.seg_r1[i] = ls.seg_r1[i];
        lg.seg_tenant[i] = ls.seg_tenant[i];
        lg.seg_tile0[i] = tiles;
        tiles += (ls.seg_r1[i] - ls.seg_r0[i] + gemm::BM - 1) / gemm::BM;
    }
    lg.seg_tile0[ls.n_seg] = tiles;
    CUtensorMap ta, tb;
    bool ok = make_tmap_bf16(&ta, A, p.M, p.K, lda, gemm::BM, gemm::BK) &&
              make_tmap_bf16(&tb, B, p.N, p.K, ldb, gemm::BN, gemm::BK) &&
              make_tmap_bf16(&lg.tt, ls.t, p.M, ls.ldt, ls.ldt, gemm::BM, 16, 32);
    for (int i = 0; i < ls.n_parts && ok; ++i) {
        lg.part_cols[i] = ls.cols[i];
        ok = make_tmap_bf16(&lg.tb[i], ls.b[i], (uint64_t)ls.n_tenants * ls.cols[i], kLoraRank,
                            kLoraRank, gemm::BN, 16, 32);
    }
    if (!ok) return fail(JNX_ERR_CUDA, "gemm: LoRA tensor map encode failed");
    const int total = tiles * (p.N / gemm::BN);
    if (total == 0) return JNX_OK;
    int grid = num_sms();
    if (total < grid) grid = total;
    if (p.group_m <= 0) p.group_m = default_group_m(p.K);
    cudaError_t e = p.epi == EPI_ROPE ? launch_epi<EPI_ROPE, true>(ta, tb, lg, p, grid, s)
                                      : launch_epi<EPI_RESID, true>(ta, tb, lg, p, grid, s);
    if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "gemm launch: %s", cudaGetErrorString(e));
    return JNX_OK;
}

}  // namespace jnx
