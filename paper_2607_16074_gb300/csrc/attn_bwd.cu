// Attention backward on the 5th-generation tensor cores (tcgen05, sm_103a):
// the gradients of the per-sample bidirectional attention (one sample's
// tokens attend to each other only), for the per-tenant LoRA backward.
//
// With S = q k^T / sqrt(hd), P = softmax(S) (rows), O = P v and the
// incoming dO:  dv = P^T dO,  dP = dO v^T,  dS = P * (dP - D) with
// D = rowsum(dO * O),  dq = dS k / sqrt(hd),  dk = dS^T q / sqrt(hd).
// P is recomputed from the forward's saved log2-sum-exp of each row, so no
// row max or normalisation is needed here.
//
// One kernel template k_attn_bwd<HD, MODE> runs one pass:
//   DQ   outer tile = 128 queries of head h, inner loop over the sample's
//        64-key tiles:       S = Q K^T, dP = dO V^T, dS, dQ += dS K
//   DKV  outer tile = 128 keys of K/V head g, inner loop over (query head
//        of the group, 64-query tile):  S^T = K Q^T, dP^T = V dO^T, P^T,
//        dS^T, dK += dS^T Q, dV += P^T dO       (head dims 64 / 128)
//   DK   as DKV without dV; DV as DKV without dP and dK (head dim 256,
//        whose two 256-column accumulators do not fit TMEM together)
// Each pass accumulates in TMEM and writes its rows once, so no atomics and
// a fixed summation order: a sample's gradients do not depend on where it
// sits in the packed batch.
//
// Warp roles (192 threads, one CTA per SM, persistent over work items):
//   warp 0     TMA producer: the item's outer operands (A1, and A2 when the
//              pass has a dP product) into one buffer, inner operands B1 /
//              B2 through rings that run on from item to item
//   warp 1     MMA issuer: the two score-shaped products of inner tile j
//              into score buffer j % 2 (S at column 64 b, dP at 128 + 64 b),
//              issued two tiles ahead of the accumulating products, which
//              read P / dS (bf16, written by the elementwise warps over the
//              first 32 columns of the buffer they came from) as the TMEM A
//              operand and the inner tile from shared memory as the MN-major
//              B operand, into the accumulator(s) at column 256
//   warps 2-5  elementwise (one outer row per thread): P = 2^(S c - lse),
//              dS = P (dP - D); then the epilogue: scale, inverse RoPE for
//              dq / dk, bf16, store
// Operands by pass:          A1   A2   B1   B2   accumulating products
//   DQ                       Q    dO   K_j  V_j  dQ += dS B1
//   DKV / DK / DV            K    V    Q_j  dO_j dK += dS^T B1, dV += P^T B2
// Rows of a tile past the sample's end hold other rows' data (or the
// tensor's zero fill): their scores are finite, their probabilities are set
// to zero through lse = +inf (inner columns) or an explicit mask (DQ keys),
// and their gradient rows are never stored.
#include <algorithm>

#include "jnx_bwd.h"
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

namespace abwd {
constexpr int BM = 128;  // outer rows per item
constexpr int BN = 64;   // inner rows per tile
enum { DQ = 0, DKV = 1, DK = 2, DV = 3 };
constexpr int kBars = 19;
}  // namespace abwd

template <int HD, int MODE>
struct AttnBwdCfg {
    static_assert(HD == 64 || HD == 128 || HD == 256, "head dim 64, 128 or 256");
    static constexpr bool NEED_DP = MODE != abwd::DV;
    static constexpr int NACC = MODE == abwd::DKV ? 2 : 1;
    static constexpr int BM = abwd::BM, BN = abwd::BN;
    static constexpr int OB = BM * HD * 2;  // one outer operand tile
    static constexpr int IB = BN * HD * 2;  // one inner operand tile
    static constexpr int NB1 = HD == 256 ? 2 : 3;
    static constexpr int NB2 = (HD == 256 && NEED_DP) ? 1 : 2;
    static constexpr int OFF_A2 = OB;
    static constexpr int OFF_B1 = NEED_DP ? 2 * OB : OB;
    static constexpr int OFF_B2 = OFF_B1 + NB1 * IB;
    static constexpr int OFF_BAR = OFF_B2 + NB2 * IB;
    static constexpr int SMEM = OFF_BAR + abwd::kBars * 8 + 16 + 1024;
    static constexpr uint32_t S_COL = 0;        // score buffer b at b * BN
    static constexpr uint32_t DP_COL = 2 * BN;  // dP buffer b at 2 BN + b * BN
    static constexpr uint32_t ACC_COL = 256;
    static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
    static_assert(ACC_COL + NACC * HD <= 512, "TMEM columns");
    static_assert(MODE != abwd::DKV || HD <= 128, "dK and dV together need head dim <= 128");
};

struct BwdItems {
    const int2* list;  // (sample, 128-row tile), most expensive first
    int n;
};

struct BwdWork {
    int tile, hp, start, L;
    bool valid;
};

// Item w: list entry w / HP, head (query head for DQ, K/V head otherwise) w % HP.
__device__ __forceinline__ BwdWork bwd_fetch(const BwdItems& it, const int* __restrict__ cu, int HP,
                                             int w, int n_work) {
    BwdWork a{0, 0, 0, 0, false};
    if (w >= n_work) return a;
    a.hp = w % HP;
    const int2 e = it.list[w / HP];
    a.tile = e.y;
    a.start = cu[e.x];
    a.L = cu[e.x + 1] - a.start;
    a.valid = a.tile * abwd::BM < a.L;
    return a;
}

template <int HD, int MODE>
__global__ void __launch_bounds__(192, 1)
    k_attn_bwd(const __grid_constant__ CUtensorMap t_qkv_o, const __grid_constant__ CUtensorMap t_qkv_i,
               const __grid_constant__ CUtensorMap t_do_o, const __grid_constant__ CUtensorMap t_do_i,
               const int* __restrict__ cu, BwdItems items, int H, int Hkv, float scale_log2,
               float scale, const float* __restrict__ lse, const float* __restrict__ Dsum,
               const int* __restrict__ pos, const float2* __restrict__ rope, int rope_ld,
               uint16_t* __restrict__ dqkv, int ldq, int* status) {
    using C = AttnBwdCfg<HD, MODE>;
    constexpr int BM = C::BM, BN = C::BN;
    constexpr int NCH = HD / 64;  // 64-column (128-byte) chunks of an operand row
    constexpr bool IS_DQ = MODE == abwd::DQ;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* sA1 = sm;
    uint8_t* sA2 = sm + C::OFF_A2;
    auto sB1 = [&](int b) { return sm + C::OFF_B1 + b * C::IB; };
    auto sB2 = [&](int b) { return sm + C::OFF_B2 + b * C::IB; };
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
    uint64_t* o_full = bars + 0;
    uint64_t* o_empty = bars + 1;
    uint64_t* b1_full = bars + 2;   // [3]
    uint64_t* b1_empty = bars + 5;  // [3]
    uint64_t* b2_full = bars + 8;   // [2]
    uint64_t* b2_empty = bars + 10; // [2]
    uint64_t* s_full = bars + 12;   // [2]
    uint64_t* p_full = bars + 14;   // [2]
    uint64_t* acc_full = bars + 16;
    uint64_t* acc_free = bars + 17;
    uint64_t* drain = bars + 18;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + abwd::kBars);
    volatile int* fail_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int group = H / Hkv;
    const int HP = IS_DQ ? H : Hkv;
    const int n_work = items.n * HP;
    if (tid == 0) {
        for (int i = 0; i < abwd::kBars; ++i)
            mbar_init(&bars[i], (i == 14 || i == 15 || i == 17) ? BM : 1);
        *fail_flag = 0;
        fence_barrier_init();
        fence_proxy_async();
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot;
    // inner tiles of an item
    auto n_inner = [&](int L) { return IS_DQ ? (L + BN - 1) / BN : group * ((L + BN - 1) / BN); };

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            tma_prefetch_desc(&t_qkv_o);
            tma_prefetch_desc(&t_qkv_i);
            tma_prefetch_desc(&t_do_o);
            tma_prefetch_desc(&t_do_i);
            bool ok = true;
            int no = 0;              // outer tiles loaded
            uint32_t g1 = 0, g2 = 0;  // inner tiles loaded into each ring
            auto load_inner = [&](const CUtensorMap* map, uint8_t* dst, int col, int row,
                                  uint64_t* full) {
                mbar_arrive_expect_tx(full, C::IB);
#pragma unroll
                for (int c = 0; c < NCH; ++c) tma_load_2d(dst + c * BN * 128, map, col + c * 64, row, full);
            };
            for (int w = blockIdx.x; w < n_work && ok && !*fail_flag; w += gridDim.x) {
                const BwdWork a = bwd_fetch(items, cu, HP, w, n_work);
                if (!a.valid) continue;
                const int row0 = a.start + a.tile * BM;
                if (no > 0 && !(ok = mbar_wait(o_empty, (no - 1) & 1))) break;
                mbar_arrive_expect_tx(o_full, C::NEED_DP ? 2 * C::OB : C::OB);
                if (IS_DQ) {
#pragma unroll
                    for (int c = 0; c < NCH; ++c) {
                        tma_load_2d(sA1 + c * BM * 128, &t_qkv_o, a.hp * HD + c * 64, row0, o_full);
                        tma_load_2d(sA2 + c * BM * 128, &t_do_o, a.hp * HD + c * 64, row0, o_full);
                    }
                } else {
#pragma unroll
                    for (int c = 0; c < NCH; ++c) {
                        tma_load_2d(sA1 + c * BM * 128, &t_qkv_o, (H + a.hp) * HD + c * 64, row0,
                                    o_full);
                        if (C::NEED_DP)
                            tma_load_2d(sA2 + c * BM * 128, &t_qkv_o, (H + Hkv + a.hp) * HD + c * 64,
                                        row0, o_full);
                    }
                }
                ++no;
                const int n = n_inner(a.L);
                const int nq = (a.L + BN - 1) / BN;
                for (int j = 0; j < n && ok; ++j) {
                    int row, c1, c2;
                    const CUtensorMap* m2;
                    if (IS_DQ) {
                        const int g = a.hp / group;
                        row = a.start + j * BN;
                        c1 = (H + g) * HD;
                        c2 = (H + Hkv + g) * HD;
                        m2 = &t_qkv_i;
                    } else {
                        const int hq = a.hp * group + j / nq;
                        row = a.start + (j % nq) * BN;
                        c1 = hq * HD;
                        c2 = hq * HD;
                        m2 = &t_do_i;
                    }
                    const int s1 = g1 % C::NB1;
                    if (!(ok = mbar_wait(&b1_empty[s1], ((g1 / C::NB1) & 1) ^ 1))) break;
                    load_inner(&t_qkv_i, sB1(s1), c1, row, &b1_full[s1]);
                    ++g1;
                    const int s2 = g2 % C::NB2;
                    if (!(ok = mbar_wait(&b2_empty[s2], ((g2 / C::NB2) & 1) ^ 1))) break;
                    load_inner(m2, sB2(s2), c2, row, &b2_full[s2]);
                    ++g2;
                }
            }
            if (!ok) *fail_flag = 1;
            // teardown: every copy issued has landed before the CTA exits
            if (no > 0) mbar_wait(o_full, (no - 1) & 1, 100000000LL);
            for (uint32_t k = 0; k < (uint32_t)C::NB1 && k < g1; ++k) {
                const uint32_t i = g1 - 1 - k;
                mbar_wait(&b1_full[i % C::NB1], (i / C::NB1) & 1, 100000000LL);
            }
            for (uint32_t k = 0; k < (uint32_t)C::NB2 && k < g2; ++k) {
                const uint32_t i = g2 - 1 - k;
                mbar_wait(&b2_full[i % C::NB2], (i / C::NB2) & 1, 100000000LL);
            }
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
            constexpr uint32_t IDESC_ACC = idesc_bf16_f32(BM, HD) | (1u << 16);  // B MN-major
            bool ok = true, issued = false;
            int no = 0;
            uint32_t c1s = 0, c2s = 0;  // B1 / B2 tiles taken by the score products
            uint32_t c1a = 0, c2a = 0;  // B1 / B2 tiles taken by the accumulating products
            uint32_t gs = 0, gp = 0;    // score tiles issued / P tiles consumed
            int items_done = 0;
            const uint32_t a1 = smem_u32(sA1), a2 = smem_u32(sA2);
            auto issue_scores = [&]() -> bool {
                const int s1 = c1s % C::NB1;
                if (!mbar_wait(&b1_full[s1], (c1s / C::NB1) & 1)) return false;
                tc_fence_after();
                const uint32_t b1 = smem_u32(sB1(s1));
                const uint32_t d = tbase + C::S_COL + (gs & 1) * BN;
#pragma unroll
                for (int ks = 0; ks < HD / 16; ++ks)
                    tc_mma_f16(d, sw128_desc(a1 + (ks >> 2) * BM * 128 + (ks & 3) * 32),
                               sw128_desc(b1 + (ks >> 2) * BN * 128 + (ks & 3) * 32), IDESC_S, ks > 0);
                if (MODE == abwd::DV) tc_commit(&b1_empty[s1]);
                ++c1s;
                if (C::NEED_DP) {
                    const int s2 = c2s % C::NB2;
                    if (!mbar_wait(&b2_full[s2], (c2s / C::NB2) & 1)) return false;
                    tc_fence_after();
                    const uint32_t b2 = smem_u32(sB2(s2));
                    const uint32_t d2 = tbase + C::DP_COL + (gs & 1) * BN;
#pragma unroll
                    for (int ks = 0; ks < HD / 16; ++ks)
                        tc_mma_f16(d2, sw128_desc(a2 + (ks >> 2) * BM * 128 + (ks & 3) * 32),
                                   sw128_desc(b2 + (ks >> 2) * BN * 128 + (ks & 3) * 32), IDESC_S,
                                   ks > 0);
                    if (MODE == abwd::DQ || MODE == abwd::DK) tc_commit(&b2_empty[s2]);
                    ++c2s;
                }
                tc_commit(&s_full[gs & 1]);
                ++gs;
                issued = true;
                return true;
            };
            // acc += X(tmem, 128 x 64 bf16) . B(smem inner tile, MN-major)
            auto acc_mma = [&](uint32_t acc_col, uint32_t xa, uint8_t* b, bool accumulate) {
                const uint32_t ba = smem_u32(b);
#pragma unroll
                for (int ks = 0; ks < BN / 16; ++ks)  // 16 inner rows = 8 TMEM columns of X
                    tc_mma_f16_ts(tbase + acc_col, xa + ks * 8,
                                  sw128_desc_mn(ba + ks * 16 * 128, BN * 128, 1024), IDESC_ACC,
                                  accumulate || ks > 0);
            };
            for (int w = blockIdx.x; w < n_work && ok && !*fail_flag; w += gridDim.x) {
                const BwdWork a = bwd_fetch(items, cu, HP, w, n_work);
                if (!a.valid) continue;
                const int n = n_inner(a.L);
                if (!(ok = mbar_wait(o_full, no & 1))) break;
                ++no;
                tc_fence_after();
                ok = issue_scores() && (n < 2 || issue_scores());
                if (ok && n <= 2) tc_commit(o_empty);
                for (int kt = 0; kt < n && ok; ++kt) {
                    const uint32_t pb = gp & 1;
                    if (!(ok = mbar_wait(&p_full[pb], (gp >> 1) & 1))) break;
                    ++gp;
                    // the first accumulating product of an item overwrites the
                    // accumulator: the previous item's epilogue must have read it
                    if (kt == 0 && items_done > 0 &&
                        !(ok = mbar_wait(acc_free, (items_done - 1) & 1)))
                        break;
                    tc_fence_after();
                    const uint32_t sb = tbase + C::S_COL + pb * BN;
                    const uint32_t db = tbase + C::DP_COL + pb * BN;
                    if (MODE == abwd::DQ || MODE == abwd::DK) {
                        const int s1 = c1a % C::NB1;
                        acc_mma(C::ACC_COL, sb, sB1(s1), kt > 0);  // dS (over S) . B1
                        tc_commit(&b1_empty[s1]);
                        ++c1a;
                    } else if (MODE == abwd::DV) {
                        const int s2 = c2a % C::NB2;
                        if (!(ok = mbar_wait(&b2_full[s2], (c2a / C::NB2) & 1))) break;
                        tc_fence_after();
                        acc_mma(C::ACC_COL, sb, sB2(s2), kt > 0);  // P^T (over S) . dO
                        tc_commit(&b2_empty[s2]);
                        ++c2a;
                    } else {  // DKV
                        const int s1 = c1a % C::NB1, s2 = c2a % C::NB2;
                        acc_mma(C::ACC_COL, db, sB1(s1), kt > 0);       // dS^T (over dP) . Q
                        acc_mma(C::ACC_COL + HD, sb, sB2(s2), kt > 0);  // P^T (over S) . dO
                        tc_commit(&b1_empty[s1]);
                        tc_commit(&b2_empty[s2]);
                        ++c1a;
                        ++c2a;
                    }
                    // the score products of tile kt + 2 reuse buffer pb: the
                    // tensor core runs this thread's MMAs in issue order, so
                    // the products above have read it before they land
                    if (kt + 2 < n) {
                        ok = issue_scores();
                        if (ok && kt + 3 == n) tc_commit(o_empty);
                    }
                }
                if (!ok) break;
                tc_commit(acc_full);
                ++items_done;
            }
            if (!ok) *fail_flag = 1;
            if (issued) {
                tc_commit(drain);
                mbar_wait(drain, 0, 100000000LL);
            }
        }
    } else {
        // ---------------- elementwise + epilogue ----------------
        const int quarter = warp & 3;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        uint32_t gs = 0;
        int items_done = 0;
        bool ok = true;
        for (int w = blockIdx.x; w < n_work && ok; w += gridDim.x) {
            if (__any_sync(0xffffffffu, *fail_flag != 0)) break;
            const BwdWork a = bwd_fetch(items, cu, HP, w, n_work);
            if (!a.valid) continue;
            const int L = a.L, n = n_inner(L);
            const int nq = (L + BN - 1) / BN;
            const int r = a.tile * BM + quarter * 32 + lane;  // this thread's outer row
            const bool rv = r < L;
            float lse_r = INFINITY, d_r = 0.f;
            if (IS_DQ && rv) {
                lse_r = lse[(size_t)(a.start + r) * H + a.hp];
                d_r = Dsum[(size_t)(a.start + r) * H + a.hp];
            }
            for (int j = 0; j < n; ++j) {
                // DKV / DK / DV: the tile's 64 query columns' lse and D, two
                // per lane, broadcast with shuffles below
                float la = INFINITY, lb = INFINITY, da = 0.f, db = 0.f;
                if (!IS_DQ) {
                    const int hq = a.hp * group + j / nq;
                    const int q0 = (j % nq) * BN;
                    if (q0 + lane < L) {
                        la = lse[(size_t)(a.start + q0 + lane) * H + hq];
                        if (C::NEED_DP) da = Dsum[(size_t)(a.start + q0 + lane) * H + hq];
                    }
                    if (q0 + 32 + lane < L) {
                        lb = lse[(size_t)(a.start + q0 + 32 + lane) * H + hq];
                        if (C::NEED_DP) db = Dsum[(size_t)(a.start + q0 + 32 + lane) * H + hq];
                    }
                }
                if (!(ok = __all_sync(0xffffffffu, mbar_wait(&s_full[gs & 1], (gs >> 1) & 1))))
                    break;
                tc_fence_after();
                const uint32_t tS = tbase + lane_base + C::S_COL + (gs & 1) * BN;
                const uint32_t tP = tbase + lane_base + C::DP_COL + (gs & 1) * BN;
                const int kvalid = L - j * BN;  // DQ: keys of this tile inside the sample
                uint32_t pk[32], dk[32];
                // one 32-column half of the S (and dP) row at a time
#pragma unroll
                for (int c = 0; c < 2; ++c) {
                    uint32_t sv[32], dv[32];
                    tmem_ld32(tS + c * 32, sv);
                    if (C::NEED_DP) tmem_ld32(tP + c * 32, dv);
                    tmem_ld_wait();
#pragma unroll
                    for (int e = 0; e < 32; e += 2) {
                        float p[2], ds[2];
#pragma unroll
                        for (int u = 0; u < 2; ++u) {
                            const int col = c * 32 + e + u;
                            const float sc_s = __uint_as_float(sv[e + u]);
                            float l, dd = 0.f;
                            if (IS_DQ) {
                                l = lse_r;
                                dd = d_r;
                            } else {
                                l = __shfl_sync(0xffffffffu, c == 0 ? la : lb, e + u);
                                if (C::NEED_DP) dd = __shfl_sync(0xffffffffu, c == 0 ? da : db, e + u);
                            }
                            p[u] = ex2_approx(sc_s * scale_log2 - l);
                            if (IS_DQ && col >= kvalid) p[u] = 0.f;
                            ds[u] = C::NEED_DP ? p[u] * (__uint_as_float(dv[e + u]) - dd) : 0.f;
                        }
                        pk[c * 16 + e / 2] = pack_bf2(p[0], p[1]);
                        dk[c * 16 + e / 2] = pack_bf2(ds[0], ds[1]);
                    }
                }
                if (MODE == abwd::DQ || MODE == abwd::DK) {
                    tmem_st32(tS, dk);
                } else if (MODE == abwd::DV) {
                    tmem_st32(tS, pk);
                } else {
                    tmem_st32(tS, pk);
                    tmem_st32(tP, dk);
                }
                tmem_st_wait();
                tc_fence_before();
                mbar_arrive(&p_full[gs & 1]);
                ++gs;
            }
            if (!ok) break;
            // ---- epilogue: the accumulator rows -> dqkv (bf16) ----
            if (!(ok = __all_sync(0xffffffffu, mbar_wait(acc_full, items_done & 1)))) break;
            tc_fence_after();
            const int grow = a.start + r;
            const uint32_t tacc = tbase + lane_base + C::ACC_COL;
            for (int acc = 0; acc < C::NACC; ++acc) {
                // which gradient: dq (DQ), dk (DK, DKV first), dv (DV, DKV second)
                const bool is_v = MODE == abwd::DV || acc == 1;
                const int colo = IS_DQ ? a.hp * HD : (is_v ? (H + Hkv + a.hp) * HD : (H + a.hp) * HD);
                const float sc = is_v ? 1.f : scale;
                const uint32_t ta = tacc + acc * HD;
                if (!is_v) {
                    // a position outside the (cos, sin) table is reported
                    // and read as position 0 (no rotation)
                    int pr = rv ? pos[grow] : 0;
                    if (pr < 0 || pr >= rope_ld) {
                        if (rv) report(status, JNX_ERR_DEVICE_BOUNDS);
                        pr = 0;
                    }
#pragma unroll 1
                    for (int c = 0; c < HD / 64; ++c) {
                        float2 cs[32];
                        if (rv) {
                            const float2* src = rope + (size_t)(c * 32) * rope_ld + pr;
#pragma unroll
                            for (int e = 0; e < 32; ++e) cs[e] = __ldg(src + (size_t)e * rope_ld);
                        }
                        uint32_t lo[32], hi[32];
                        tmem_ld32(ta + c * 32, lo);
                        tmem_ld32(ta + HD / 2 + c * 32, hi);
                        tmem_ld_wait();
                        if (rv) {
                            uint32_t plo[16], phi[16];
#pragma unroll
                            for (int e = 0; e < 32; e += 2) {
                                float x[2], y[2];
#pragma unroll
                                for (int u = 0; u < 2; ++u) {
                                    const float a0 = sc * __uint_as_float(lo[e + u]);
                                    const float b0 = sc * __uint_as_float(hi[e + u]);
                                    x[u] = a0 * cs[e + u].x + b0 * cs[e + u].y;
                                    y[u] = b0 * cs[e + u].x - a0 * cs[e + u].y;
                                }
                                plo[e / 2] = pack_bf2(x[0], x[1]);
                                phi[e / 2] = pack_bf2(y[0], y[1]);
                            }
                            uint4* olo = reinterpret_cast<uint4*>(dqkv + (size_t)grow * ldq + colo + c * 32);
                            uint4* ohi = reinterpret_cast<uint4*>(dqkv + (size_t)grow * ldq + colo +
                                                                  HD / 2 + c * 32);
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                olo[u] = make_uint4(plo[4 * u], plo[4 * u + 1], plo[4 * u + 2], plo[4 * u + 3]);
                                ohi[u] = make_uint4(phi[4 * u], phi[4 * u + 1], phi[4 * u + 2], phi[4 * u + 3]);
                            }
                        }
                    }
                } else {
#pragma unroll 1
                    for (int c = 0; c < HD / 32; ++c) {
                        uint32_t v[32];
                        tmem_ld32(ta + c * 32, v);
                        tmem_ld_wait();
                        if (rv) {
                            uint4* o = reinterpret_cast<uint4*>(dqkv + (size_t)grow * ldq + colo + c * 32);
#pragma unroll
                            for (int u = 0; u < 4; ++u)
                                o[u] = make_uint4(pack_bf2(__uint_as_float(v[8 * u]), __uint_as_float(v[8 * u + 1])),
                                                  pack_bf2(__uint_as_float(v[8 * u + 2]), __uint_as_float(v[8 * u + 3])),
                                                  pack_bf2(__uint_as_float(v[8 * u + 4]), __uint_as_float(v[8 * u + 5])),
                                                  pack_bf2(__uint_as_float(v[8 * u + 6]), __uint_as_float(v[8 * u + 7])));
                        }
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(acc_free);
            ++items_done;
        }
        if (!ok) *fail_flag = 1;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (*fail_flag && tid == 0) report(status, JNX_ERR_TIMEOUT);
    if (warp == 1) tmem_dealloc(tbase, 512);
}

template <int HD, int MODE>
static jnx_status launch_bwd(const CUtensorMap (&maps)[4], const int* cu, const BwdItems& it, int H,
                             int Hkv, const float* lse, const float* D, const int* pos,
                             const float2* rope, int rope_ld, uint16_t* dqkv, int ldq, int* status,
                             cudaStream_t s) {
    using C = AttnBwdCfg<HD, MODE>;
    static std::atomic<uint64_t> attr{0};
    if (set_smem_limit(reinterpret_cast<const void*>(k_attn_bwd<HD, MODE>), C::SMEM, attr) !=
        cudaSuccess)
        return fail(JNX_ERR_CUDA, "attention backward: smem attribute");
    const int HP = MODE == abwd::DQ ? H : Hkv;
    const long long n_work = (long long)it.n * HP;
    if (n_work > 0x7FFFFFFFLL) return fail(JNX_ERR_UNSUPPORTED, "attention backward: too many items");
    if (n_work == 0) return JNX_OK;
    const int grid = (int)std::min<long long>(n_work, num_sms());
    const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
    const float scale = (float)(1.0 / sqrt((double)HD));
    k_attn_bwd<HD, MODE><<<grid, 192, C::SMEM, s>>>(maps[0], maps[1], maps[2], maps[3], cu, it, H,
                                                   Hkv, scale_log2, scale, lse, D, pos, rope,
                                                   rope_ld, dqkv, ldq, status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK
                            : fail(JNX_ERR_CUDA, "attention backward: %s", cudaGetErrorString(e));
}

jnx_status attention_bwd_launch(const uint16_t* qkv, int ldq, const uint16_t* dO, const float* lse,
                                const float* D, int n_tokens, int H, int Hkv, int hd,
                                const int* cu, const int* pos, const float2* rope, int rope_ld,
                                const int2* items, int n_items, uint16_t* dqkv, int* status,
                                cudaStream_t s) {
    if (n_tokens == 0 || n_items == 0) return JNX_OK;
    if (!items) return fail(JNX_ERR_INVALID_ARG, "attention backward: null work items");
    if (Hkv <= 0 || H % Hkv) return fail(JNX_ERR_UNSUPPORTED, "attention backward: H %% Hkv != 0");
    if (ldq != (H + 2 * Hkv) * hd)
        return fail(JNX_ERR_INVALID_ARG, "attention backward: q|k|v row stride");
    CUtensorMap maps[4];
    if (!make_tmap_bf16(&maps[0], qkv, n_tokens, ldq, ldq, abwd::BM, 64) ||
        !make_tmap_bf16(&maps[1], qkv, n_tokens, ldq, ldq, abwd::BN, 64) ||
        !make_tmap_bf16(&maps[2], dO, n_tokens, (uint64_t)H * hd, (uint64_t)H * hd, abwd::BM, 64) ||
        !make_tmap_bf16(&maps[3], dO, n_tokens, (uint64_t)H * hd, (uint64_t)H * hd, abwd::BN, 64))
        return fail(JNX_ERR_CUDA, "attention backward: tensor map encode failed");
    BwdItems it{items, n_items};
    jnx_status st;
    switch (hd) {
        case 64:
            if ((st = launch_bwd<64, abwd::DQ>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld, dqkv,
                                               ldq, status, s)))
                return st;
            return launch_bwd<64, abwd::DKV>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld, dqkv,
                                             ldq, status, s);
        case 128:
            if ((st = launch_bwd<128, abwd::DQ>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld,
                                                dqkv, ldq, status, s)))
                return st;
            return launch_bwd<128, abwd::DKV>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld, dqkv,
                                              ldq, status, s);
        case 256:
            if ((st = launch_bwd<256, abwd::DQ>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld,
                                                dqkv, ldq, status, s)) ||
                (st = launch_bwd<256, abwd::DK>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld,
                                                dqkv, ldq, status, s)))
                return st;
            return launch_bwd<256, abwd::DV>(maps, cu, it, H, Hkv, lse, D, pos, rope, rope_ld, dqkv,
                                             ldq, status, s);
        default:
            return fail(JNX_ERR_UNSUPPORTED, "attention backward: head_dim %d", hd);
    }
}

}  // namespace jnx
