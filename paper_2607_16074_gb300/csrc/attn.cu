// Varlen attention confined to each sample (block-diagonal, bidirectional).
//
// Every sample is one observation prefix; its tokens attend to each other
// and to nothing else, so the kernels only visit (sample, 128-query tile,
// head) triples inside a sample and the key loop only walks that sample's
// keys: no cross-sample tile is ever computed.  Tiles start at the sample's
// first token, so a sample's result is the same wherever it sits in the
// packed batch (grouped == isolated).
//
// One tcgen05 kernel, k_attn_ws: S, P and O live in TMEM, Q/K/V arrive by
// TMA; persistent and warp-specialised, with two independent streams of
// query tiles per CTA for head dims 64 / 128 and one for head dim 256 (whose
// O accumulator leaves no TMEM for a second stream).
// Q, K, V come from the fused projection output [N, (H + 2 Hkv) hd]; query
// head h reads K/V head h / (H / Hkv) (MQA when Hkv = 1).
#include "jnx_dev.cuh"
#include "jnx_kernels.h"

namespace jnx {

// ---------------------------------------------------------------------------
// Persistent warp-specialised tcgen05 attention (head dims 64 / 128 / 256).
//
// One CTA per SM runs NST independent streams of work items (two for head
// dims 64 / 128, one for 256); an item is one 128-query tile of one sample
// and head, and its key loop walks that sample's keys in BN-key tiles.
// Stream t owns
//   warp t        TMA producer: Q (one buffer, refilled as soon as the
//                 item's last S MMA has completed), K and V through
//                 separate 2-deep rings that run on from item to item
//   warp 2 + t    MMA issuer: S(kt) = Q K(kt)^T into one of two TMEM score
//                 buffers, O += P(kt) V(kt) into the TMEM accumulator; S runs
//                 two tiles ahead of PV, so the tensor core computes the next
//                 scores while the softmax warps work on the current ones
//   warps 4 + 8t + 4h + q (h = 0, 1; q = 0..3)
//                 online softmax and epilogue: two warpgroups, each thread
//                 holding one query row (lane 32 q + lane) and half of each
//                 64-key score tile (columns 32 h .. 32 h + 31); the two
//                 threads of a row exchange their half-row max every tile and
//                 their partial row sums in the epilogue, and each normalises
//                 and stores half of O's columns
// and TMEM columns from 256 t: S buffers at +0 and +BN, O (HD columns) at
// +2 BN.  P (bf16, two per 32-bit column) overwrites the first BN / 2
// columns of the score buffer it was computed from and is the TMEM A
// operand of the PV MMA; V is read from shared memory as the MN-major B
// operand.  With two score buffers P is double-buffered too, so the softmax
// of tile kt does not wait for PV(kt-1) (only a rare rescale of O does).
// The two streams share nothing but the tensor core, so one stream's
// softmax overlaps the other's MMAs and copies, and a short tail tile costs
// only its own stream.  P of half 1 (keys 32..63) lands in score columns
// 16..31, which hold half 0's scores: it is written only after the row's
// exchange, which half 0 reaches after its scores are in registers.
//
// The running max is lazy: a row raises the max m it subtracts only when a
// new tile's max exceeds it by more than 8 (log2 units), so O is rarely
// rescaled; the probabilities stay below 2^8 and O / l does not depend on m.
//
// Barriers per stream (each role tracks parities with completion counters):
//   q_full, q_empty          Q landed / the item's last S MMA completed
//   k_full[2], k_empty[2]    K ring (a slot frees when its S MMA completes)
//   v_full[2], v_empty[2]    V ring (a slot frees when its PV MMA completes)
//   s_full[2]                score buffer b holds a new S
//   p_full[2]                P of a tile written over its S in score
//                            buffer b (256 arrivals: both halves)
//   o_done[2]                PV of a tile with score buffer b completed; a
//                            softmax thread waits for PV(g-2) before it
//                            arrives for tile g, so neither barrier runs two
//                            phases ahead of a waiter
//   o_free                   the epilogue has read O (256 arrivals)
//   drain                    all MMAs of the stream completed (teardown)
//   xbar[4][2]               exchange between the two threads of each row:
//                            per lane quarter q and slot (exchange count % 2),
//                            64 arrivals (the warp pair); the exchanged
//                            values live in a [slot][half][row] array, a slot
//                            reused two exchanges later, after the partner
//                            has passed the next exchange (every wait, as
//                            all of them, bounded)
// ---------------------------------------------------------------------------
namespace attn_ws {
constexpr int BM = 128;        // query rows per item
constexpr float kLazy = 8.0f;  // log2 growth of the max that forces a rescale
constexpr int kBars = 18;      // barriers per stream
}  // namespace attn_ws

// Work items: an explicit (sample, query tile) list, or, without one, every
// (sample, query tile) combination sample-major (a sample's query tiles,
// which read the same K/V, run close together) with the empty ones skipped.
struct AttnItems {
    const int2* list;
    int n;      // entries of `list`, or S * tiles
    int tiles;  // query tiles per sample in the enumeration (longest sample)
};

// One work item: query tile qt of the sample at packed rows [start,
// start + L), head h.  Fetched one item ahead by every role so that the
// list and cu_seqlens loads of the next item overlap the current one.
struct AttnWork {
    int qt, h, start, L;
    bool valid;  // false past the end, or for an empty enumerated item
};

__device__ __forceinline__ AttnWork attn_fetch(const AttnItems& it, const int* __restrict__ cu,
                                               int H, int w, int n_work) {
    AttnWork a{0, 0, 0, 0, false};
    if (w >= n_work) return a;
    a.h = w % H;
    const int i = w / H;
    int s;
    if (it.list) {
        const int2 e = it.list[i];
        s = e.x;
        a.qt = e.y;
    } else {
        a.qt = i % it.tiles;
        s = i / it.tiles;
    }
    a.start = cu[s];
    a.L = cu[s + 1] - a.start;
    a.valid = a.qt * attn_ws::BM < a.L;
    return a;
}

// Epilogue staging of 16 output columns (32 bytes a row) through a 1 KB
// slot per softmax warp: thread `lane` puts its row's two 16-byte units;
// in round i thread `lane` gets row 16 i + lane / 2, unit lane % 2, so each
// store instruction writes 16 rows x 32 contiguous bytes.  Units are
// XOR-swizzled by (row / 4) % 2 (no bank conflicts either way).
__device__ __forceinline__ void attn_stg_put(uint8_t* stg, int lane, const uint4 (&v)[2]) {
    uint8_t* rowp = stg + lane * 32;
    const int sw = (lane >> 2) & 1;
    *reinterpret_cast<uint4*>(rowp + ((0 ^ sw) << 4)) = v[0];
    *reinterpret_cast<uint4*>(rowp + ((1 ^ sw) << 4)) = v[1];
}

__device__ __forceinline__ uint4 attn_stg_get(const uint8_t* stg, int lane, int i) {
    const int r = 16 * i + (lane >> 1), j = lane & 1;
    return *reinterpret_cast<const uint4*>(stg + r * 32 + ((j ^ ((r >> 2) & 1)) << 4));
}

template <int HD, int BN>
struct AttnWsCfg {
    static_assert(BN == 64, "key tile of 64 keys");
    static_assert(HD == 64 || HD == 128 || HD == 256, "head dim 64, 128 or 256");
    // streams per CTA: a stream holds two BN-column score buffers and an
    // HD-column O in TMEM (512 columns), so head dim 256 runs one stream
    static constexpr int NST = HD == 256 ? 1 : 2;
    // softmax warpgroups per stream: each takes half of a tile's columns
    // (and half of O's columns in the epilogue) for all 128 rows
    static constexpr int SPLIT = 2;
    static constexpr int HCOLS = BN / SPLIT;   // score columns per softmax thread
    static constexpr int SMW = 4 * SPLIT * NST;  // softmax warps
    static constexpr int THREADS = 128 + 32 * SMW;
    static constexpr uint32_t TSTRIDE = 256;  // TMEM columns between streams
    static constexpr int BM = attn_ws::BM;
    static constexpr int QB = BM * HD * 2;  // Q tile
    static constexpr int KB = BN * HD * 2;  // one K (or V) tile
    static constexpr int OFF_K = QB;
    static constexpr int OFF_V = OFF_K + 2 * KB;
    static constexpr int STREAM = OFF_V + 2 * KB;  // bytes per stream (multiple of 1024)
    static constexpr int OFF_STG = NST * STREAM;  // epilogue staging, 1 KB per softmax warp
    // row-max / row-sum exchange between a stream's two halves:
    // [stream][slot 0/1][half][BM] floats
    static constexpr int OFF_XM = OFF_STG + SMW * 1024;
    static constexpr int OFF_BAR = OFF_XM + NST * 2 * SPLIT * BM * 4;
    static constexpr int NBAR = attn_ws::kBars + 8;  // + exchange barriers [quarter][slot]
    static constexpr int SMEM = OFF_BAR + NST * NBAR * 8 + 16 + 1024;
    static_assert(STREAM % 1024 == 0, "128B-swizzled tiles need 1024-byte alignment");
    static_assert(SMEM <= 227 * 1024, "shared memory per CTA");
    static constexpr uint32_t O_COL = 2 * BN;  // within the stream's 256 columns
    static_assert(O_COL + HD <= (NST == 2 ? TSTRIDE : 512), "TMEM columns per stream");
};

// Softmax of one 128 x 64 score tile, split between two threads per row:
// this thread holds 32 of the row's scores (v) and kvalid of them lie in
// the sample (FULL: all 32).  attn_half_max: the raw max of the valid ones;
// attn_half_exp: p = 2^(s scale - m) packed as bf16 pairs, and their sum.
// The exponential of one key pair in four: ex2_poly2 (jnx_dev.cuh), which
// takes load off the MUFU pipe the softmax warps share.
template <bool FULL>
__device__ __forceinline__ float attn_half_max(const uint32_t (&v)[32], int kvalid) {
    float mx4[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) mx4[j] = -INFINITY;
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
        const float a0 = __uint_as_float(v[e]), a1 = __uint_as_float(v[e + 1]);
        float& acc = mx4[(e >> 1) & 3];
        if (FULL) {
            acc = fmax3(acc, a0, a1);
        } else {
            if (e < kvalid) acc = fmaxf(acc, a0);
            if (e + 1 < kvalid) acc = fmaxf(acc, a1);
        }
    }
    return fmax3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3]));
}

template <bool FULL>
__device__ __forceinline__ void attn_half_exp(const uint32_t (&v)[32], int kvalid,
                                              float scale_log2, float m, float& rs,
                                              uint32_t (&pk)[16]) {
    const uint64_t sc2 = f2_pack(scale_log2, scale_log2), nm2 = f2_pack(-m, -m);
    uint64_t rs2[2] = {f2_pack(0.f, 0.f), f2_pack(0.f, 0.f)};
#pragma unroll
    for (int e = 0; e < 32; e += 2) {
        float x0, x1;
        f2_unpack(f2_fma(f2_pack(__uint_as_float(v[e]), __uint_as_float(v[e + 1])), sc2, nm2),
                  x0, x1);
        float p0, p1;
        if (FULL && ((e >> 1) & 3) == 3) {
            ex2_poly2(x0, x1, p0, p1);
        } else {
            p0 = ex2_approx(x0);
            p1 = ex2_approx(x1);
        }
        if (!FULL) {
            if (e >= kvalid) p0 = 0.f;
            if (e + 1 >= kvalid) p1 = 0.f;
        }
        rs2[(e >> 1) & 1] = f2_add(rs2[(e >> 1) & 1], f2_pack(p0, p1));
        pk[e / 2] = pack_bf2(p0, p1);
    }
    float r0, r1, r2, r3;
    f2_unpack(rs2[0], r0, r1);
    f2_unpack(rs2[1], r2, r3);
    rs = (r0 + r1) + (r2 + r3);
}

template <int HD, int BN>
__global__ void __launch_bounds__(HD == 256 ? 384 : 640, 1)
    k_attn_ws(const __grid_constant__ CUtensorMap tq, const __grid_constant__ CUtensorMap tkv,
              const int* __restrict__ cu, AttnItems items, int H, int Hkv, float scale_log2,
              uint16_t* __restrict__ out, int ldo, float* __restrict__ lse, int* status) {
    using C = AttnWsCfg<HD, BN>;
    constexpr int BM = C::BM;
    constexpr int NCH = HD / 64;  // 64-column (128-byte) chunks of a Q/K/V row
    extern __shared__ uint8_t smem_raw[];
    uint8_t* sm = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(sm + C::OFF_BAR + C::NST * C::NBAR * 8);
    volatile int* fail_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // stream of this warp: producers 0/1, MMA issuers 2/3, then per stream
    // 4 SPLIT softmax warps (stream t, half h, lane quarter q: warp
    // 4 + 4 SPLIT t + 4 h + q, so warp % 4 = q)
    const int t = warp < 4 ? (warp & 1) : (warp - 4) / (4 * C::SPLIT);
    uint8_t* st = sm + t * C::STREAM;
    uint8_t* sQ = st;
    auto sK = [&](int b) { return st + C::OFF_K + b * C::KB; };
    auto sV = [&](int b) { return st + C::OFF_V + b * C::KB; };
    uint64_t* bars = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR) + t * C::NBAR;
    uint64_t* q_full = bars + 0;
    uint64_t* q_empty = bars + 1;
    uint64_t* k_full = bars + 2;   // [2]
    uint64_t* k_empty = bars + 4;  // [2]
    uint64_t* v_full = bars + 6;   // [2]
    uint64_t* v_empty = bars + 8;  // [2]
    uint64_t* s_full = bars + 10;  // [2]
    uint64_t* p_full = bars + 12;  // [2]
    uint64_t* o_done = bars + 14;  // [2]
    uint64_t* o_free = bars + 16;
    uint64_t* drain = bars + 17;
    uint64_t* xbar = bars + attn_ws::kBars;  // [quarter][slot]: the halves' exchanges

    const int n_work = items.n * H;
    const int group = H / Hkv;
    const int w0 = C::NST * blockIdx.x + t, dw = C::NST * gridDim.x;
    if (tid == 0) {
        // both streams' barriers: one arrival each, but p_full[] and o_free,
        // which every softmax thread of the stream arrives on, and the
        // exchange barriers, which the 64 threads of a warp pair arrive on
        uint64_t* all = reinterpret_cast<uint64_t*>(sm + C::OFF_BAR);
        for (int i = 0; i < C::NST * C::NBAR; ++i) {
            const int k = i % C::NBAR;
            mbar_init(&all[i], k >= attn_ws::kBars                  ? 64
                               : (k == 12 || k == 13 || k == 16) ? C::SPLIT * BM
                                                                 : 1);
        }
        *fail_flag = 0;
        fence_barrier_init();
        fence_proxy_async();
    }
    if (warp == 2) {
        tmem_alloc(tmem_slot, 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tmem_slot + (uint32_t)t * C::TSTRIDE;

    if (warp < 2) {
        // ---------------- producer of stream t ----------------
        if (lane == 0 && t < C::NST) {
            tma_prefetch_desc(&tq);
            tma_prefetch_desc(&tkv);
            bool ok = true;
            int nq = 0;            // Q tiles loaded
            uint32_t gk = 0, gv = 0;  // K / V tiles loaded
            auto load_kv = [&](bool is_v, uint32_t& g, int y, int col) -> bool {
                const int b = g & 1;
                uint64_t* full = is_v ? &v_full[b] : &k_full[b];
                if (!mbar_wait(is_v ? &v_empty[b] : &k_empty[b], ((g >> 1) & 1) ^ 1)) return false;
                mbar_arrive_expect_tx(full, C::KB);
                uint8_t* dst = is_v ? sV(b) : sK(b);
#pragma unroll
                for (int c = 0; c < NCH; ++c)
                    tma_load_2d(dst + c * BN * 128, &tkv, col + c * 64, y, full);
                ++g;
                return true;
            };
            AttnWork nxt = attn_fetch(items, cu, H, w0, n_work);
            for (int w = w0; w < n_work && ok && !*fail_flag; w += dw) {
                const AttnWork a = nxt;
                nxt = attn_fetch(items, cu, H, w + dw, n_work);
                if (!a.valid) continue;
                const int start = a.start, L = a.L, qt = a.qt, h = a.h;
                const int n_kt = (L + BN - 1) / BN;
                const int kvh = h / group;
                if (nq > 0 && !(ok = mbar_wait(q_empty, (nq - 1) & 1))) break;
                mbar_arrive_expect_tx(q_full, C::QB);
#pragma unroll
                for (int c = 0; c < NCH; ++c)
                    tma_load_2d(sQ + c * BM * 128, &tq, h * HD + c * 64, start + qt * BM, q_full);
                ++nq;
                // K runs one tile ahead of V: S(kt + 1) is issued before PV(kt)
                for (int j = 0; j <= n_kt && ok; ++j) {
                    if (j < n_kt) ok = load_kv(false, gk, start + j * BN, (H + kvh) * HD);
                    if (ok && j > 0)
                        ok = load_kv(true, gv, start + (j - 1) * BN, (H + Hkv + kvh) * HD);
                }
            }
            if (!ok) *fail_flag = 1;
            // teardown: every copy this thread issued has landed before the
            // CTA may exit (immediate in a normal run: the MMA warp has
            // consumed them all)
            if (nq > 0) mbar_wait(q_full, (nq - 1) & 1);
            for (uint32_t k = 0; k < 2 && k < gk; ++k)
                mbar_wait(&k_full[(gk - 1 - k) & 1], ((gk - 1 - k) >> 1) & 1);
            for (uint32_t k = 0; k < 2 && k < gv; ++k)
                mbar_wait(&v_full[(gv - 1 - k) & 1], ((gv - 1 - k) >> 1) & 1);
        }
    } else if (warp < 4) {
        // ---------------- MMA issuer of stream t ----------------
        if (lane == 0 && t < C::NST) {
            constexpr uint32_t IDESC_S = idesc_bf16_f32(BM, BN);
            constexpr uint32_t IDESC_PV = idesc_bf16_f32(BM, HD) | (1u << 16);  // B MN-major
            bool ok = true, issued = false;
            int nq = 0;                  // Q tiles consumed
            uint32_t gk = 0, gv = 0;     // K / V tiles consumed
            uint32_t gs = 0;             // S tiles issued (score buffer gs & 1)
            uint32_t gp = 0;             // p_full completions consumed = PVs issued
            int items_done = 0;
            auto issue_s = [&](const uint32_t qa) -> bool {
                const int b = gk & 1;
                if (!mbar_wait(&k_full[b], (gk >> 1) & 1)) return false;
                tc_fence_after();
                const uint32_t ka = smem_u32(sK(b));
                const uint32_t d = tbase + (gs & 1) * BN;
#pragma unroll
                for (int ks = 0; ks < HD / 16; ++ks)
                    tc_mma_f16(d, sw128_desc(qa + (ks >> 2) * BM * 128 + (ks & 3) * 32),
                               sw128_desc(ka + (ks >> 2) * BN * 128 + (ks & 3) * 32), IDESC_S,
                               ks > 0);
                tc_commit(&s_full[gs & 1]);
                tc_commit(&k_empty[b]);
                ++gk;
                ++gs;
                issued = true;
                return true;
            };
            AttnWork nxt = attn_fetch(items, cu, H, w0, n_work);
            for (int w = w0; w < n_work && ok && !*fail_flag; w += dw) {
                const AttnWork a = nxt;
                nxt = attn_fetch(items, cu, H, w + dw, n_work);
                if (!a.valid) continue;
                const int n_kt = (a.L + BN - 1) / BN;
                if (!(ok = mbar_wait(q_full, nq & 1))) break;
                ++nq;
                tc_fence_after();
                const uint32_t qa = smem_u32(sQ);
                // S(0), S(1): their score buffers were read before the
                // previous item's last PVs were issued
                ok = issue_s(qa) && (n_kt < 2 || issue_s(qa));
                if (ok && n_kt <= 2) tc_commit(q_empty);
                for (int kt = 0; kt < n_kt && ok; ++kt) {
                    // P(kt) is in TMEM, over S(kt) in score buffer gp & 1
                    const uint32_t pb = gp & 1;
                    if (!(ok = mbar_wait(&p_full[pb], (gp >> 1) & 1))) break;
                    ++gp;
                    // the first PV of an item overwrites O: the previous
                    // item's epilogue must have read it
                    if (kt == 0 && items_done > 0 && !(ok = mbar_wait(o_free, (items_done - 1) & 1)))
                        break;
                    const int b = gv & 1;
                    if (!(ok = mbar_wait(&v_full[b], (gv >> 1) & 1))) break;
                    tc_fence_after();
                    const uint32_t pa = tbase + pb * BN, va = smem_u32(sV(b));
#pragma unroll
                    for (int ks = 0; ks < BN / 16; ++ks)  // 16 keys = 8 TMEM columns of P
                        tc_mma_f16_ts(tbase + C::O_COL, pa + ks * 8,
                                      sw128_desc_mn(va + ks * 16 * 128, BN * 128, 1024), IDESC_PV,
                                      kt > 0 || ks > 0);
                    tc_commit(&o_done[pb]);
                    tc_commit(&v_empty[b]);
                    ++gv;
                    // S(kt + 2) reuses the score buffer of S(kt) / P(kt): the
                    // tensor core runs this thread's MMAs in issue order, so
                    // PV(kt) has read P(kt) before S(kt + 2) lands there
                    if (kt + 2 < n_kt) {
                        ok = issue_s(qa);
                        if (ok && kt + 3 == n_kt) tc_commit(q_empty);
                    }
                }
                ++items_done;
            }
            if (!ok) *fail_flag = 1;
            if (issued) {
                tc_commit(drain);
                mbar_wait(drain, 0);
            }
        }
    } else {
        // ---------------- softmax + epilogue of stream t ----------------
        // This thread: row quarter * 32 + lane of the item's query tile,
        // score columns [32 half, 32 half + 32) of each key tile, O columns
        // [HD/2 half, HD/2 half + HD/2) in the epilogue.
        const int quarter = warp & 3;  // TMEM lanes this warp may access
        const int half = ((warp - 4) >> 2) % C::SPLIT;
        const int row = quarter * 32 + lane;
        const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
        const uint32_t tO = tbase + lane_base + C::O_COL + half * (HD / 2);
        float* xm = reinterpret_cast<float*>(sm + C::OFF_XM) + t * 2 * C::SPLIT * BM;
        uint32_t gs = 0;  // S tiles consumed
        uint32_t nw = 0;  // PVs this thread has seen complete (in order)
        uint32_t xg = 0;  // exchanges with the other half
        // wait until PV(0 .. upto-1) of this stream have completed
        auto wait_pv = [&](uint32_t upto) -> bool {
            for (; nw < upto; ++nw)
                if (!__all_sync(0xffffffffu, mbar_wait(&o_done[nw & 1], (nw >> 1) & 1)))
                    return false;
            tc_fence_after();
            return true;
        };
        // exchange a value with the thread of the other half that holds the
        // same row (slot xg % 2 of the shared array, a 64-arrival barrier of
        // the warp pair; the slot is rewritten two exchanges later, after
        // the partner has passed the next exchange, i.e. read this one).
        // The fences order this thread's TMEM loads before the partner's
        // stores past the barrier (the partner's P overwrites scores).
        auto exchange = [&](float mine, float& other) -> bool {
            const int slot = xg & 1;
            float* x = xm + slot * C::SPLIT * BM;
            x[half * BM + row] = mine;
            tc_fence_before();
            mbar_arrive(&xbar[quarter * 2 + slot]);
            const bool got =
                __all_sync(0xffffffffu, mbar_wait(&xbar[quarter * 2 + slot], (xg >> 1) & 1));
            tc_fence_after();
            other = x[(half ^ 1) * BM + row];
            ++xg;
            return got;
        };
        bool ok = true;
        AttnWork nxt = attn_fetch(items, cu, H, w0, n_work);
        for (int w = w0; w < n_work && ok; w += dw) {
            if (__any_sync(0xffffffffu, *fail_flag != 0)) break;
            const AttnWork a = nxt;
            if (!a.valid) {
                nxt = attn_fetch(items, cu, H, w + dw, n_work);
                continue;
            }
            const int start = a.start, L = a.L, qt = a.qt, h = a.h;
            const int n_kt = (L + BN - 1) / BN;
            float m = 0.f, l = 0.f;  // running max (shared by the halves); this half's row sum
            for (int kt = 0; kt < n_kt; ++kt) {
                // waits are made warp-uniform: TMEM loads are warp-collective
                if (!(ok = __all_sync(0xffffffffu, mbar_wait(&s_full[gs & 1], (gs >> 1) & 1))))
                    break;
                tc_fence_after();
                const uint32_t tS = tbase + lane_base + (gs & 1) * BN;
                const uint32_t g = gs++;  // stream-wide index of this tile
                const int kvalid = L - kt * BN - half * C::HCOLS;  // of this half's keys
                const bool full = L - kt * BN >= BN;
                uint32_t v[32];
                tmem_ld32(tS + half * C::HCOLS, v);
                tmem_ld_wait();
                float mine = full ? attn_half_max<true>(v, kvalid) : attn_half_max<false>(v, kvalid);
                float theirs;
                if (!(ok = exchange(mine, theirs))) break;
                const float mx = fmaxf(mine, theirs) * scale_log2;
                float alpha = 1.f;
                if (kt == 0) {
                    m = mx;
                } else if (mx > m + attn_ws::kLazy) {
                    alpha = ex2_approx(m - mx);
                    m = mx;
                }
                uint32_t pk[16];
                float rs;
                if (full)
                    attn_half_exp<true>(v, kvalid, scale_log2, m, rs, pk);
                else
                    attn_half_exp<false>(v, kvalid, scale_log2, m, rs, pk);
                if (kt > 0 && __any_sync(0xffffffffu, alpha < 1.f)) {
                    // rescaling O needs every earlier PV of the item done;
                    // each half rescales its half of O's columns
                    if (!(ok = wait_pv(g))) break;
#pragma unroll 1
                    for (int c = 0; c < HD / 2 / 16; ++c) {
                        uint32_t o16[16];
                        tmem_ld16(tO + c * 16, o16);
                        tmem_ld_wait();
#pragma unroll
                        for (int e = 0; e < 16; ++e)
                            o16[e] = __float_as_uint(__uint_as_float(o16[e]) * alpha);
                        tmem_st16(tO + c * 16, o16);
                    }
                    tmem_st_wait();
                }
                l = l * alpha + rs;
                // keeps o_done[b] within one phase of this thread's waits
                if (g >= 2 && !(ok = wait_pv(g - 1))) break;
                // P of this half's 32 keys: 16 columns of bf16 pairs, over
                // the score buffer's first 32 columns (keys in order)
                tmem_st16(tS + half * (C::HCOLS / 2), pk);
                tmem_st_wait();
                tc_fence_before();
                mbar_arrive(&p_full[g & 1]);
            }
            if (!ok) break;
            // the next item's loads overlap this epilogue (fetched here, not
            // at the top, so they hold no registers during the key loop)
            nxt = attn_fetch(items, cu, H, w + dw, n_work);
            // epilogue: O / l -> bf16 once the item's last PV is done; the
            // row sum is the two halves' sums, added in half order
            if (!(ok = wait_pv(gs))) break;
            float lo;
            if (!(ok = exchange(l, lo))) break;
            const float ltot = half == 0 ? l + lo : lo + l;
            const float inv = 1.0f / ltot;
            if (half == 0 && lse != nullptr && qt * BM + row < L)
                lse[(size_t)(start + qt * BM + row) * H + h] = m + log2f(ltot);
            // 16 columns at a time through this warp's staging slot; O is
            // released (o_free) once its last columns are in registers
            uint8_t* stg = sm + C::OFF_STG + (warp - 4) * 1024;
            const int row0 = qt * BM + quarter * 32;  // first row of this warp
            constexpr int NCK = HD / 2 / 16;            // 16-column chunks of this half
            uint32_t ov[2][16];
            tmem_ld16(tO, ov[0]);
#pragma unroll
            for (int c = 0; c < NCK; ++c) {
                uint32_t(&v)[16] = ov[c & 1];
                tmem_ld_wait_regs16(v);
                if (c + 1 < NCK) {
                    tmem_ld16(tO + (c + 1) * 16, ov[(c + 1) & 1]);
                } else {
                    tc_fence_before();
                    mbar_arrive(o_free);
                }
                uint4 q2[2];
#pragma unroll
                for (int u = 0; u < 2; ++u)
                    q2[u] = make_uint4(pack_bf2(__uint_as_float(v[8 * u]) * inv,
                                                __uint_as_float(v[8 * u + 1]) * inv),
                                       pack_bf2(__uint_as_float(v[8 * u + 2]) * inv,
                                                __uint_as_float(v[8 * u + 3]) * inv),
                                       pack_bf2(__uint_as_float(v[8 * u + 4]) * inv,
                                                __uint_as_float(v[8 * u + 5]) * inv),
                                       pack_bf2(__uint_as_float(v[8 * u + 6]) * inv,
                                                __uint_as_float(v[8 * u + 7]) * inv));
                attn_stg_put(stg, lane, q2);
                __syncwarp();
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const int rr = 16 * i + (lane >> 1);
                    const uint4 w4 = attn_stg_get(stg, lane, i);
                    if (row0 + rr < L)
                        *reinterpret_cast<uint4*>(out + (size_t)(start + row0 + rr) * ldo + h * HD +
                                                  half * (HD / 2) + c * 16 + (lane & 1) * 8) = w4;
                }
                __syncwarp();
            }
        }
        if (!ok) *fail_flag = 1;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (*fail_flag && tid == 0) report(status, JNX_ERR_TIMEOUT);
    if (warp == 2) tmem_dealloc(*tmem_slot, 512);
}

template <int HD, int BN>
static jnx_status launch_attn_ws(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv,
                                 const int* cu, int S, int max_seqlen, const int2* items,
                                 int n_items, uint16_t* out, int ldo, float* lse, int* status,
                                 cudaStream_t s) {
    using C = AttnWsCfg<HD, BN>;
    static std::atomic<uint64_t> attr{0};
    if (set_smem_limit(reinterpret_cast<const void*>(k_attn_ws<HD, BN>), C::SMEM, attr) !=
        cudaSuccess)
        return fail(JNX_ERR_CUDA, "attention: smem attribute");
    CUtensorMap tq, tkv;
    if (!make_tmap_bf16(&tq, qkv, n_tokens, ldq, ldq, C::BM, 64) ||
        !make_tmap_bf16(&tkv, qkv, n_tokens, ldq, ldq, BN, 64))
        return fail(JNX_ERR_CUDA, "attention: tensor map encode failed");
    AttnItems it;
    it.tiles = (max_seqlen + C::BM - 1) / C::BM;
    if (items) {
        it.list = items;
        it.n = n_items;
    } else {
        it.list = nullptr;
        it.n = S * it.tiles;
    }
    if ((long long)it.n * H > 0x7FFFFFFFLL)
        return fail(JNX_ERR_UNSUPPORTED, "attention: too many work items");
    const int n_work = it.n * H;
    if (n_work == 0) return JNX_OK;
    const int grid = std::min((n_work + C::NST - 1) / C::NST, num_sms());
    const float scale_log2 = (float)(1.4426950408889634 / sqrt((double)HD));
    k_attn_ws<HD, BN><<<grid, C::THREADS, C::SMEM, s>>>(tq, tkv, cu, it, H, Hkv, scale_log2, out, ldo,
                                                 lse, status);
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "attention: %s", cudaGetErrorString(e));
}

jnx_status attention_launch(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv, int hd,
                            const int* cu, int S, int max_seqlen, const int2* items, int n_items,
                            uint16_t* out, int ldo, float* lse, int* status, cudaStream_t s) {
    if (S == 0 || max_seqlen == 0) return JNX_OK;
    if (Hkv <= 0 || H % Hkv) return fail(JNX_ERR_UNSUPPORTED, "attention: H %% Hkv != 0");
    if ((long long)S * ((max_seqlen + attn_ws::BM - 1) / attn_ws::BM) > 0x7FFFFFFFLL || H > 65535)
        return fail(JNX_ERR_UNSUPPORTED, "attention: grid too large");
    switch (hd) {
        case 64:
            return launch_attn_ws<64, 64>(qkv, ldq, n_tokens, H, Hkv, cu, S, max_seqlen, items,
                                          n_items, out, ldo, lse, status, s);
        case 128:
            return launch_attn_ws<128, 64>(qkv, ldq, n_tokens, H, Hkv, cu, S, max_seqlen, items,
                                           n_items, out, ldo, lse, status, s);
        case 256:
            return launch_attn_ws<256, 64>(qkv, ldq, n_tokens, H, Hkv, cu, S, max_seqlen, items,
                                           n_items, out, ldo, lse, status, s);
        default:
            return fail(JNX_ERR_UNSUPPORTED, "attention: head_dim %d not in {64,128,256}", hd);
    }
}

}  // namespace jnx
