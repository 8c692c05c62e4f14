// jnx_backbone_backward_lora: the gradients of every group tenant's loss with
// respect to that tenant's own LoRA adapters, back through the frozen shared
// backbone (tenant-private backward, §5.2 and App. A; adapters as the
// tenant's lightweight module, §3.1).
//
// Memory plan (GB300-first): the forward keeps only each block's fp32
// residual input (jnx_backbone_forward_train); the backward recomputes one
// block at a time from it (its activations then live in one block-sized
// workspace) and runs that block's backward right away, so the full 2B-class
// group's activations are never all resident at once.
//
// Per block, with dy = dloss/d(block output) (fp32) and its bf16 copy:
//   recompute   n1 = RMSNorm(x), t = n1 A^T, q|k|v = RoPE(n1 W_qkv^T + t B^T),
//               O = Attn (+ its log2-sum-exp), h = x + O W_o^T (+ adapter),
//               n2 = RMSNorm(h)
//   FFN         dm = dy W_down (bf16, into the up columns of the packed
//               gate/up buffer); the gate/up GEMM recomputed from n2 with
//               dg = dm u act'(g), du = dm act(g) in its epilogue (in place
//               over dm); dn2 = [dg|du] W_gu; dh = dy + RMSNorm'(h; dn2)
//   O           dO = dh W_o + (dh B_o) A_o;  dB_o = dh^T t_o, dA_o = (dh B_o)^T O
//   attention   dq, dk, dv (tcgen05 passes, inverse RoPE on dq, dk)
//   Q/K/V       dB = dY^T t, dA = (dY B)^T n1, dn1 = dqkv W_qkv + sum (dY B) A;
//               dx = dh + RMSNorm'(x; dn1)  -> dy of the block below
// Input-gradient GEMMs read transposed copies of the frozen weights
// (jnx_layer_t), so every product is the library's K-major tcgen05 GEMM.
#include <algorithm>
#include <vector>

#include "../../include/jnx_ops.h"
#include "jnx_bwd.h"
#include "jnx_dev.cuh"
#include "jnx_kernels.h"
#include "jnx_trace.h"

using namespace jnx;

namespace {

constexpr size_t kAlign = 256;
size_t up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

struct BwdWs {
    int* status;
    float *xh, *dy, *dh, *dn, *datt, *lse, *Dsum, *part;
    uint16_t *dy_bf, *dh_bf, *n1, *n2, *qkv, *dqkv, *att, *dO, *gu;
    uint16_t *t_qkv, *t_o, *dt_qkv, *dt_o, *bt[4];
    float2* rope;
    int2* items;
    size_t part_floats;
    size_t bytes;
};

// The GLU's backward with its gate/up GEMM recomputed: dm [M, F] = dy
// W_down^T (W_down^T stored as wdt [F, d]) goes, bf16, into the up columns
// of gu [M, 2F] (packed order: 128-column blocks alternating gate and up);
// the gate/up GEMM over the normed rows n2 [M, d] then leaves dg = dm u
// act'(g) in the gate columns and du = dm act(g) in the up columns.  Each
// up column is read by the tile that writes it, so no other buffer is
// needed.
jnx_status ffn_glu_backward(const uint16_t* dy_bf, const uint16_t* wdt, const uint16_t* n2,
                                   const uint16_t* w_gu, int64_t M, int64_t F, int64_t d, int act,
                                   uint16_t* gu, int* status, cudaStream_t s) {
    jnx_status st;
    GemmParams p{};
    p.M = (int)M;
    p.N = (int)F;
    p.K = (int)d;
    p.epi = EPI_BF16;
    p.pack_up = 1;
    p.out = gu;
    p.ldo = (int)(2 * F);
    p.status = status;
    {
        TraceScope ts(JNX_K_GEMM_BWD, 2.0 * M * F * d, s);
        if ((st = gemm_launch(dy_bf, (int)d, wdt, (int)d, p, s))) return st;
    }
    p = GemmParams{};
    p.M = (int)M;
    p.N = (int)(2 * F);
    p.K = (int)d;
    p.epi = EPI_GLU_DM;
    p.out = gu;
    p.ldo = (int)(2 * F);
    p.aux = gu;
    p.ldaux = (int)(2 * F);
    p.act = act;
    p.status = status;
    TraceScope ts(JNX_K_GEMM_GU, 2.0 * M * 2.0 * F * d, s);
    return gemm_launch(n2, (int)d, w_gu, (int)d, p, s);
}

BwdWs carve_bwd(const jnx_backbone* bb, int64_t N, void* base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    BwdWs w{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* r = p ? p + off : nullptr;
        off += up(bytes);
        return r;
    };
    const size_t d = bb->d_model, H = bb->n_heads, Hkv = bb->n_kv_heads, hd = bb->head_dim;
    const size_t qkvw = (H + 2 * Hkv) * hd, F = bb->d_ff, T = std::max(bb->n_tenants, 1);
    const size_t n = (size_t)std::max<int64_t>(N, 1);
    auto f32 = [&](size_t cnt) { return reinterpret_cast<float*>(take(cnt * 4)); };
    auto b16 = [&](size_t cnt) { return reinterpret_cast<uint16_t*>(take(cnt * 2)); };
    w.status = reinterpret_cast<int*>(take(256));
    w.xh = f32(n * d);
    w.dy = f32(n * d);
    w.dh = f32(n * d);
    w.dn = f32(n * d);
    w.datt = f32(n * H * hd);
    w.lse = f32(n * H);
    w.Dsum = f32(n * H);
    w.part_floats = seg_tn_part_floats((int)n, kSegMaxSlots, (int)std::max(d, H * hd));
    w.part = f32(w.part_floats);
    w.dy_bf = b16(n * d);
    w.dh_bf = b16(n * d);
    w.n1 = b16(n * d);
    w.n2 = b16(n * d);
    w.qkv = b16(n * qkvw);
    w.dqkv = b16(n * qkvw);
    w.att = b16(n * H * hd);
    w.dO = b16(n * H * hd);
    w.gu = b16(n * 2 * F);
    w.t_qkv = b16(n * 3 * kLoraRank);
    w.t_o = b16(n * kLoraRank);
    w.dt_qkv = b16(n * 3 * kLoraRank);
    w.dt_o = b16(n * kLoraRank);
    const size_t cols[4] = {H * hd, Hkv * hd, Hkv * hd, d};
    for (int i = 0; i < 4; ++i) w.bt[i] = b16(T * kLoraRank * cols[i]);
    w.rope = reinterpret_cast<float2*>(take((size_t)kMaxRopePos * (hd / 2) * 8));
    w.items = reinterpret_cast<int2*>(take((n + n / 128 + 1) * sizeof(int2)));
    w.bytes = off;
    return w;
}

jnx_status cuda_ok(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

}  // namespace

extern "C" size_t jnx_backbone_backward_workspace_bytes(const jnx_backbone* bb, int32_t n_tokens) {
    if (!bb || n_tokens < 0) return 0;
    return carve_bwd(bb, n_tokens, nullptr).bytes;
}

extern "C" jnx_status jnx_transpose(const uint16_t* src, int32_t batch, int32_t rows, int32_t cols,
                                    uint16_t* dst, void* stream) {
    clear_error();
    if ((!src || !dst) && (size_t)batch * rows * cols > 0)
        return fail(JNX_ERR_INVALID_ARG, "transpose: null buffer");
    if (src == dst && batch > 0 && rows > 0 && cols > 0)
        return fail(JNX_ERR_INVALID_ARG, "transpose: in place");
    return transpose_launch(src, batch, rows, cols, dst, static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_backbone_backward_lora(const jnx_backbone* bb, const jnx_layer_t* lt,
                                                 const jnx_group* g, const float* saved,
                                                 const float* d_hidden,
                                                 const jnx_lora_grads* grads, int32_t accumulate,
                                                 void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    jnx_status st;
    if ((st = check_backbone(bb)) || (st = check_group(g))) return st;
    if (bb->lora_rank != kLoraRank)
        return fail(JNX_ERR_INVALID_ARG, "backward: the backbone has no rank-%d adapters", kLoraRank);
    if (!lt || !saved || !d_hidden || !grads || !workspace)
        return fail(JNX_ERR_INVALID_ARG, "backward: null argument");
    const int N = g->n_tokens, d = bb->d_model, H = bb->n_heads, Hkv = bb->n_kv_heads,
              hd = bb->head_dim, F = bb->d_ff, T = bb->n_tenants;
    const int qkvw = (H + 2 * Hkv) * hd, Hhd = H * hd;
    const int cols[4] = {Hhd, Hkv * hd, Hkv * hd, d};
    const int offs[3] = {0, Hhd, Hhd + Hkv * hd};
    if (d % 256 || Hhd % 256 || (Hkv * hd) % 256)
        return fail(JNX_ERR_UNSUPPORTED, "backward: widths must be multiples of 256");
    for (int l = 0; l < bb->n_layers; ++l) {
        const jnx_layer_t& t = lt[l];
        const jnx_lora_grads& gr = grads[l];
        if (!t.w_qkv_t || !t.w_o_t || !t.w_gu_t || !t.w_down_t)
            return fail(JNX_ERR_INVALID_ARG, "backward: layer %d has a null transposed weight", l);
        if (!gr.a_q || !gr.b_q || !gr.a_k || !gr.b_k || !gr.a_v || !gr.b_v || !gr.a_o || !gr.b_o)
            return fail(JNX_ERR_INVALID_ARG, "backward: layer %d has a null gradient buffer", l);
    }
    if (g->n_slots > std::min(kSegMaxSlots, kLoraMaxSlots))
        return fail(JNX_ERR_UNSUPPORTED, "backward: groups hold at most %d tenants",
                    std::min(kSegMaxSlots, kLoraMaxSlots));
    for (int i = 0; i < g->n_slots; ++i)
        if (g->h_slot_tenant[i] < 0 || g->h_slot_tenant[i] >= T)
            return fail(JNX_ERR_INVALID_ARG, "backward: tenant %d has no adapter",
                        g->h_slot_tenant[i]);
    BwdWs w = carve_bwd(bb, N, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "backward: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    if (N == 0) return JNX_OK;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bool add = accumulate != 0;
    const double Nd = (double)N * d;

    {
        TraceScope ts(JNX_K_ROPE_TABLE, (double)g->max_seqlen * hd * 4.0, s);
        if ((st = rope_table_launch(w.rope, g->max_seqlen, hd, bb->rope_theta, s))) return st;
    }
    int n_items = 0;
    const int2* items = nullptr;
    if ((st = attn_items_for(g, w.items, s, "backward", items, n_items))) return st;
    double attn_flops = 0.0;
    for (int i = 0; i < g->n_samples; ++i) {
        const double L = g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i];
        attn_flops += 4.0 * L * L * H * hd;
    }
    std::vector<int> seg_r0, seg_r1;
    for (int i = 0; i < g->n_slots; ++i) {
        seg_r0.push_back(g->h_cu_seqlens[g->h_seg_offsets[i]]);
        seg_r1.push_back(g->h_cu_seqlens[g->h_seg_offsets[i + 1]]);
    }
    LoraSpec lq{}, lo{};
    lq.t = w.t_qkv;
    lq.ldt = 3 * kLoraRank;
    lq.n_parts = 3;
    lq.cols[0] = cols[0];
    lq.cols[1] = cols[1];
    lq.cols[2] = cols[2];
    lo.t = w.t_o;
    lo.ldt = kLoraRank;
    lo.n_parts = 1;
    lo.cols[0] = d;
    for (LoraSpec* ls : {&lq, &lo}) {
        ls->n_tenants = T;
        ls->n_seg = g->n_slots;
        ls->seg_r0 = seg_r0.data();
        ls->seg_r1 = seg_r1.data();
        ls->seg_tenant = g->h_slot_tenant;
    }
    static thread_local SegUpParts sp;

    // the final RMSNorm: dy = RMSNorm'(x_L; d_hidden)
    {
        TraceScope ts(JNX_K_NORM_BWD, Nd * 18.0, s);
        if ((st = rms_bwd_launch(saved + (size_t)bb->n_layers * N * d, bb->final_norm, bb->eps,
                                 d_hidden, nullptr, N, d, w.dy, w.dy_bf, s)))
            return st;
    }
    for (int l = bb->n_layers - 1; l >= 0; --l) {
        const jnx_layer& L = bb->layers[l];
        const jnx_layer_t& Lt = lt[l];
        const jnx_lora_grads& G = grads[l];
        const float* x = saved + (size_t)l * N * d;
        const uint16_t* A[4] = {L.lora_a_q, L.lora_a_k, L.lora_a_v, L.lora_a_o};
        const uint16_t* Bm[4] = {L.lora_b_q, L.lora_b_k, L.lora_b_v, L.lora_b_o};
        float* gA[4] = {G.a_q, G.a_k, G.a_v, G.a_o};
        float* gB[4] = {G.b_q, G.b_k, G.b_v, G.b_o};

        // ---------------- recompute the block's forward ----------------
        {
            TraceScope ts(JNX_K_RMSNORM, Nd * 6.0, s);
            if ((st = rmsnorm_launch(x, L.attn_norm, bb->eps, N, d, w.n1, s))) return st;
        }
        {
            TraceScope ts(JNX_K_LORA, 2.0 * N * d * 3 * kLoraRank, s);
            if ((st = lora_down_launch(g, w.n1, d, d, 3, A, w.t_qkv, 3 * kLoraRank, s))) return st;
        }
        GemmParams p{};
        p.M = N;
        p.N = qkvw;
        p.K = d;
        p.epi = EPI_ROPE;
        p.out = w.qkv;
        p.ldo = qkvw;
        p.pos = g->pos_ids;
        p.rope = w.rope;
        p.rope_ld = g->max_seqlen;
        p.rope_cols = (H + Hkv) * hd;
        p.hd = hd;
        p.status = w.status;
        lq.b[0] = Bm[0];
        lq.b[1] = Bm[1];
        lq.b[2] = Bm[2];
        {
            TraceScope ts(JNX_K_GEMM_QKV, 2.0 * N * qkvw * d, s);
            if ((st = gemm_launch_lora(w.n1, d, L.w_qkv, d, p, lq, s))) return st;
        }
        {
            TraceScope ts(JNX_K_ATTN, attn_flops, s);
            if ((st = attention_launch(w.qkv, qkvw, N, H, Hkv, hd, g->cu_seqlens, g->n_samples,
                                       g->max_seqlen, items, n_items, w.att, Hhd, w.lse,
                                       w.status, s)))
                return st;
        }
        if (cudaMemcpyAsync(w.xh, x, (size_t)N * d * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
            return cuda_ok("backward: residual copy");
        {
            TraceScope ts(JNX_K_LORA, 2.0 * N * Hhd * kLoraRank, s);
            if ((st = lora_down_launch(g, w.att, Hhd, Hhd, 1, &A[3], w.t_o, kLoraRank, s)))
                return st;
        }
        p = GemmParams{};
        p.M = N;
        p.N = d;
        p.K = Hhd;
        p.epi = EPI_RESID;
        p.resid = w.xh;
        p.ldr = d;
        p.status = w.status;
        lo.b[0] = Bm[3];
        {
            TraceScope ts(JNX_K_GEMM_O, 2.0 * N * d * Hhd, s);
            if ((st = gemm_launch_lora(w.att, Hhd, L.w_o, Hhd, p, lo, s))) return st;
        }
        {
            TraceScope ts(JNX_K_RMSNORM, Nd * 6.0, s);
            if ((st = rmsnorm_launch(w.xh, L.ffn_norm, bb->eps, N, d, w.n2, s))) return st;
        }
        // ---------------- feed-forward backward ----------------
        // dm = dy W_down (the gradient at act(g) * u) into the up columns of
        // gu, then the gate/up GEMM recomputed from the normed rows n2 with
        // dg = dm u act'(g) and du = dm act(g) formed in its epilogue
        if ((st = ffn_glu_backward(w.dy_bf, Lt.w_down_t, w.n2, L.w_gu, N, F, d, bb->glu, w.gu,
                                   w.status, s)))
            return st;
        p = GemmParams{};
        p.M = N;
        p.N = d;
        p.K = 2 * F;
        p.epi = EPI_F32;
        p.out = w.dn;
        p.ldo = d;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_GEMM_BWD, 2.0 * N * d * 2.0 * F, s);
            if ((st = gemm_launch(w.gu, 2 * F, Lt.w_gu_t, 2 * F, p, s))) return st;
        }
        {
            TraceScope ts(JNX_K_NORM_BWD, Nd * 18.0, s);
            if ((st = rms_bwd_launch(w.xh, L.ffn_norm, bb->eps, w.dn, w.dy, N, d, w.dh, w.dh_bf, s)))
                return st;
        }

        // ---------------- O projection backward ----------------
        p = GemmParams{};
        p.M = N;
        p.N = Hhd;
        p.K = d;
        p.epi = EPI_F32;
        p.out = w.datt;
        p.ldo = Hhd;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_GEMM_BWD, 2.0 * N * Hhd * d, s);
            if ((st = gemm_launch(w.dh_bf, d, Lt.w_o_t, d, p, s))) return st;
        }
        {
            TraceScope ts(JNX_K_LORA_BWD, 2.0 * N * kLoraRank * (3.0 * d + 2.0 * Hhd), s);
            if ((st = transpose_launch(Bm[3], T, d, kLoraRank, w.bt[3], s)) ||
                (st = lora_down_launch(g, w.dh_bf, d, d, 1, &w.bt[3], w.dt_o, kLoraRank, s)) ||
                (st = seg_tn_launch(g, w.t_o, kLoraRank, w.dh_bf, d, d, w.part, w.part_floats,
                                    gB[3], (long long)d * kLoraRank, true, add, s)) ||
                (st = seg_tn_launch(g, w.dt_o, kLoraRank, w.att, Hhd, Hhd, w.part, w.part_floats,
                                    gA[3], (long long)kLoraRank * Hhd, false, add, s)))
                return st;
            sp = SegUpParts{};
            sp.n_parts = 1;
            sp.t[0] = w.dt_o;
            sp.ldt[0] = kLoraRank;
            sp.k[0] = kLoraRank;
            seg_up_weights(g, sp, 0, A[3], (long long)kLoraRank * Hhd);
            if ((st = seg_up_launch(g, sp, Hhd, w.datt, Hhd, true, s))) return st;
        }

        // ---------------- attention backward ----------------
        {
            TraceScope ts(JNX_K_NORM_BWD, (double)N * Hhd * 8.0, s);
            if ((st = attn_bwd_prep_launch(w.datt, w.att, N, H, hd, w.dO, w.Dsum, s))) return st;
        }
        {
            TraceScope ts(JNX_K_ATTN_BWD, 2.5 * attn_flops, s);
            if ((st = attention_bwd_launch(w.qkv, qkvw, w.dO, w.lse, w.Dsum, N, H, Hkv, hd,
                                           g->cu_seqlens, g->pos_ids, w.rope, g->max_seqlen,
                                           items, n_items, w.dqkv, w.status, s)))
                return st;
        }

        // ---------------- Q / K / V projections backward ----------------
        {
            TraceScope ts(JNX_K_LORA_BWD, 2.0 * N * kLoraRank * (2.0 * qkvw + 3.0 * d), s);
            for (int q = 0; q < 3; ++q) {
                uint16_t* dtq = w.dt_qkv + q * kLoraRank;
                const uint16_t* dy_q = w.dqkv + offs[q];
                if ((st = transpose_launch(Bm[q], T, cols[q], kLoraRank, w.bt[q], s)) ||
                    (st = lora_down_launch(g, dy_q, qkvw, cols[q], 1, &w.bt[q], dtq,
                                           3 * kLoraRank, s)) ||
                    (st = seg_tn_launch(g, w.t_qkv + q * kLoraRank, 3 * kLoraRank, dy_q, qkvw,
                                        cols[q], w.part, w.part_floats, gB[q],
                                        (long long)cols[q] * kLoraRank, true, add, s)) ||
                    (st = seg_tn_launch(g, dtq, 3 * kLoraRank, w.n1, d, d, w.part, w.part_floats,
                                        gA[q], (long long)kLoraRank * d, false, add, s)))
                    return st;
            }
        }
        p = GemmParams{};
        p.M = N;
        p.N = d;
        p.K = qkvw;
        p.epi = EPI_F32;
        p.out = w.dn;
        p.ldo = d;
        p.status = w.status;
        {
            TraceScope ts(JNX_K_GEMM_BWD, 2.0 * N * d * qkvw, s);
            if ((st = gemm_launch(w.dqkv, qkvw, Lt.w_qkv_t, qkvw, p, s))) return st;
        }
        {
            TraceScope ts(JNX_K_LORA_BWD, 2.0 * N * 3.0 * kLoraRank * d, s);
            sp = SegUpParts{};
            sp.n_parts = 3;
            for (int q = 0; q < 3; ++q) {
                sp.t[q] = w.dt_qkv + q * kLoraRank;
                sp.ldt[q] = 3 * kLoraRank;
                sp.k[q] = kLoraRank;
                seg_up_weights(g, sp, q, A[q], (long long)kLoraRank * d);
            }
            if ((st = seg_up_launch(g, sp, d, w.dn, d, true, s))) return st;
        }
        {
            TraceScope ts(JNX_K_NORM_BWD, Nd * 18.0, s);
            if ((st = rms_bwd_launch(x, L.attn_norm, bb->eps, w.dn, w.dh, N, d, w.dy, w.dy_bf, s)))
                return st;
        }
    }
    return cuda_ok("backward");
}

// ---------------------------------------------------------------------------
// stage-level entry points of the backward (jnx_ops.h)
// ---------------------------------------------------------------------------

extern "C" jnx_status jnx_op_attention_lse(const uint16_t* qkv, int32_t n_tokens, int32_t n_heads,
                                           int32_t n_kv_heads, int32_t head_dim,
                                           const int32_t* cu_seqlens, int32_t n_samples,
                                           int32_t max_seqlen, uint16_t* out, float* lse,
                                           int32_t* status, void* stream) {
    clear_error();
    if (!qkv || !out || !lse || (n_samples > 0 && !cu_seqlens) || n_tokens < 0)
        return fail(JNX_ERR_INVALID_ARG, "attention: null argument");
    const int ldq = (n_heads + 2 * n_kv_heads) * head_dim;
    return attention_launch(qkv, ldq, n_tokens, n_heads, n_kv_heads, head_dim, cu_seqlens,
                            n_samples, max_seqlen, nullptr, 0, out, n_heads * head_dim, lse,
                            status, static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_op_attention_backward_prep(const float* datt, const uint16_t* att,
                                                     int32_t n_tokens, int32_t n_heads,
                                                     int32_t head_dim, uint16_t* dO, float* D,
                                                     void* stream) {
    clear_error();
    if (n_tokens > 0 && (!datt || !att || !dO || !D))
        return fail(JNX_ERR_INVALID_ARG, "attention prep: null argument");
    return attn_bwd_prep_launch(datt, att, n_tokens, n_heads, head_dim, dO, D,
                                static_cast<cudaStream_t>(stream));
}

extern "C" size_t jnx_op_attention_backward_workspace_bytes(int32_t n_tokens, int32_t max_seqlen,
                                                            int32_t head_dim) {
    if (n_tokens < 0 || max_seqlen < 0 || head_dim <= 0) return 0;
    const size_t n = (size_t)n_tokens;
    return up((size_t)std::max(max_seqlen, 1) * (head_dim / 2) * 8) +
           up((n + n / 128 + 1) * sizeof(int2));
}

extern "C" jnx_status jnx_op_attention_backward(const uint16_t* qkv, const uint16_t* dO,
                                                const float* lse, const float* D, int32_t n_tokens,
                                                int32_t n_heads, int32_t n_kv_heads,
                                                int32_t head_dim, const int32_t* cu_seqlens,
                                                const int32_t* h_cu_seqlens, int32_t n_samples,
                                                int32_t max_seqlen, const int32_t* pos,
                                                float rope_theta, uint16_t* dqkv, void* workspace,
                                                size_t ws_bytes, int32_t* status, void* stream) {
    clear_error();
    if (n_tokens < 0 || n_samples < 0 || max_seqlen < 0)
        return fail(JNX_ERR_INVALID_ARG, "attention backward: negative size");
    if (n_tokens == 0 || n_samples == 0) return JNX_OK;
    if (!qkv || !dO || !lse || !D || !cu_seqlens || !h_cu_seqlens || !pos || !dqkv || !workspace)
        return fail(JNX_ERR_INVALID_ARG, "attention backward: null argument");
    if (max_seqlen > kMaxRopePos)
        return fail(JNX_ERR_UNSUPPORTED, "attention backward: sample longer than %d", kMaxRopePos);
    if (ws_bytes < jnx_op_attention_backward_workspace_bytes(n_tokens, max_seqlen, head_dim))
        return fail(JNX_ERR_WORKSPACE, "attention backward: workspace too small");
    for (int i = 0; i < n_samples; ++i) {
        const int L = h_cu_seqlens[i + 1] - h_cu_seqlens[i];
        if (L < 0 || L > max_seqlen || h_cu_seqlens[i + 1] > n_tokens || h_cu_seqlens[0] < 0)
            return fail(JNX_ERR_INVALID_ARG, "attention backward: bad sample %d", i);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    float2* rope = static_cast<float2*>(workspace);
    int2* items_d = reinterpret_cast<int2*>(static_cast<uint8_t*>(workspace) +
                                            up((size_t)std::max(max_seqlen, 1) * (head_dim / 2) * 8));
    jnx_group g{};
    g.n_samples = n_samples;
    g.n_tokens = n_tokens;
    g.h_cu_seqlens = h_cu_seqlens;
    std::vector<int2> items;
    jnx_status st;
    if ((st = refuse_capture(s, "attention backward"))) return st;
    if ((st = build_attn_items(&g, items))) return st;
    if (!items.empty() && cudaMemcpyAsync(items_d, items.data(), items.size() * sizeof(int2),
                                          cudaMemcpyHostToDevice, s) != cudaSuccess)
        return cuda_ok("attention backward: work items");
    if ((st = rope_table_launch(rope, max_seqlen, head_dim, rope_theta, s))) return st;
    const int ldq = (n_heads + 2 * n_kv_heads) * head_dim;
    TraceScope ts(JNX_K_ATTN_BWD, 0.0, s);
    return attention_bwd_launch(qkv, ldq, dO, lse, D, n_tokens, n_heads, n_kv_heads, head_dim,
                                cu_seqlens, pos, rope, max_seqlen, items_d, (int)items.size(),
                                dqkv, status, s);
}

extern "C" jnx_status jnx_op_rms_backward(const float* x, const uint16_t* gamma, float eps,
                                          const float* dn, const float* dres, int32_t M, int32_t d,
                                          float* dx, uint16_t* dx_bf, void* stream) {
    clear_error();
    if (M > 0 && (!x || !gamma || !dn || !dx))
        return fail(JNX_ERR_INVALID_ARG, "rms backward: null argument");
    return rms_bwd_launch(x, gamma, eps, dn, dres, M, d, dx, dx_bf,
                          static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_op_ffn_glu_backward(const uint16_t* dy, const uint16_t* w_down_t,
                                              const uint16_t* n2, const uint16_t* w_gu, int32_t M,
                                              int32_t F, int32_t d, int32_t act, uint16_t* gu,
                                              void* stream) {
    clear_error();
    if (M < 0 || F <= 0 || d <= 0)
        return fail(JNX_ERR_INVALID_ARG, "ffn glu backward: bad sizes");
    if (M > 0 && (!dy || !w_down_t || !n2 || !w_gu || !gu))
        return fail(JNX_ERR_INVALID_ARG, "ffn glu backward: null argument");
    if ((reinterpret_cast<uintptr_t>(gu) & 15) || F % 256 || d % 64)
        return fail(JNX_ERR_INVALID_ARG, "ffn glu backward: gu alignment, F %% 256 or d %% 64");
    if (act != JNX_GLU_SWIGLU && act != JNX_GLU_GEGLU_TANH)
        return fail(JNX_ERR_INVALID_ARG, "ffn glu backward: unknown activation %d", act);
    return ffn_glu_backward(dy, w_down_t, n2, w_gu, M, F, d, act, gu, nullptr,
                            static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_op_gemm_glu_backward(const uint16_t* A, const uint16_t* W, int32_t M,
                                               int32_t F, int32_t K, uint16_t* gu, int32_t act,
                                               void* stream) {
    clear_error();
    if (M > 0 && (!A || !W || !gu)) return fail(JNX_ERR_INVALID_ARG, "glu backward: null argument");
    (void)act;
    if ((reinterpret_cast<uintptr_t>(gu) & 15) || F % 256)
        return fail(JNX_ERR_INVALID_ARG, "glu backward: gu alignment or F %% 256");
    GemmParams p{};
    p.M = M;
    p.N = F;
    p.K = K;
    p.epi = EPI_GLU_BWD;
    p.out = gu;
    p.ldo = 2 * F;
    p.aux = gu;
    p.ldaux = 2 * F;
    p.act = act;
    TraceScope ts(JNX_K_GEMM_BWD, 2.0 * M * F * K, static_cast<cudaStream_t>(stream));
    return gemm_launch(A, K, W, K, p, static_cast<cudaStream_t>(stream));
}
