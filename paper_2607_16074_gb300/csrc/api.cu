// C-ABI entry points: the shared backbone forward, the tenant heads, status
// and helpers, plus the stage-level entry points of jnx_ops.h.
#include <algorithm>
#include <cmath>
#include <vector>

#include "../../include/jnx_ops.h"
#include "jnx_bwd.h"
#include "jnx_dev.cuh"
#include "jnx_heads.h"
#include "jnx_kernels.h"
#include "jnx_trace.h"

using namespace jnx;

namespace {

constexpr size_t kAlign = 256;
constexpr size_t kStatusBytes = 256;

size_t up(size_t v) { return (v + kAlign - 1) / kAlign * kAlign; }

// Workspace carve-up of jnx_backbone_forward.
struct BackboneWs {
    int* status;
    float* x;         // residual stream [N, d] fp32
    uint16_t* nrm;    // GEMM input of the folded RMSNorm: bf16(x * gamma) [N, d]
    float* ss;        // its per-row, per-128-column-block sums of x^2 [N, d / 128]
    uint16_t* qkv;    // [N, (H + 2 Hkv) hd] bf16
    uint16_t* att;    // [N, H hd] bf16
    uint16_t* u;      // [N, F] bf16
    float2* rope;     // [max_pos, hd / 2]
    uint16_t* t_qkv;  // LoRA: n1 [A_q | A_k | A_v]^T  [N, 3r] bf16
    uint16_t* t_o;    // LoRA: attention output A_o^T  [N, r] bf16
    int2* attn_items; // attention work items (sample, 128-query tile)
    size_t bytes;
};

BackboneWs carve_backbone(const jnx_backbone* bb, int64_t N, void* base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    BackboneWs w{};
    const int64_t d = bb->d_model, qkvw = (int64_t)(bb->n_heads + 2 * bb->n_kv_heads) * bb->head_dim;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* r = p ? p + off : nullptr;
        off += up(bytes);
        return r;
    };
    w.status = reinterpret_cast<int*>(take(kStatusBytes));
    w.x = reinterpret_cast<float*>(take((size_t)N * d * 4));
    w.nrm = reinterpret_cast<uint16_t*>(take((size_t)N * d * 2));
    w.ss = reinterpret_cast<float*>(take((size_t)N * (d / 128) * 4));
    w.qkv = reinterpret_cast<uint16_t*>(take((size_t)N * qkvw * 2));
    w.att = reinterpret_cast<uint16_t*>(take((size_t)N * bb->n_heads * bb->head_dim * 2));
    w.u = reinterpret_cast<uint16_t*>(take((size_t)N * bb->d_ff * 2));
    w.rope = reinterpret_cast<float2*>(take((size_t)kMaxRopePos * (bb->head_dim / 2) * 8));
    if (bb->lora_rank) {
        w.t_qkv = reinterpret_cast<uint16_t*>(take((size_t)N * 3 * kLoraRank * 2));
        w.t_o = reinterpret_cast<uint16_t*>(take((size_t)N * kLoraRank * 2));
    }
    // at most one item per sample plus one per 128 tokens
    w.attn_items = reinterpret_cast<int2*>(take((size_t)(N + N / 128 + 1) * sizeof(int2)));
    w.bytes = off;
    return w;
}

jnx_status cuda_status(const char* what) {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? JNX_OK : fail(JNX_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

}  // namespace

// A call that uploads a per-group work list from host memory (the attention
// items) cannot be captured into a CUDA graph: the graph would replay the
// copy from a host buffer that is gone by then.  Refused before any launch.
jnx_status jnx::refuse_capture(cudaStream_t s, const char* what) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) {
        cudaGetLastError();
        return fail(JNX_ERR_UNSUPPORTED, "%s: cannot tell whether the stream is capturing", what);
    }
    if (cs != cudaStreamCaptureStatusNone)
        return fail(JNX_ERR_UNSUPPORTED,
                    "%s: cannot be captured into a CUDA graph (it uploads a per-group work list "
                    "from host memory)", what);
    return JNX_OK;
}

namespace jnx {

jnx_status check_backbone(const jnx_backbone* bb) {
    if (!bb || !bb->layers || !bb->text_table || !bb->final_norm)
        return fail(JNX_ERR_INVALID_ARG, "backbone: null descriptor field");
    if (bb->n_layers < 0 || bb->n_heads <= 0 || bb->n_kv_heads <= 0 ||
        bb->n_heads % bb->n_kv_heads)
        return fail(JNX_ERR_INVALID_ARG, "backbone: bad head counts");
    if (bb->head_dim != 64 && bb->head_dim != 128 && bb->head_dim != 256)
        return fail(JNX_ERR_UNSUPPORTED, "backbone: head_dim %d not in {64,128,256}", bb->head_dim);
    const int d = bb->d_model;
    if (d != 256 && d != 512 && d != 1024 && d != 2048 && d != 4096)
        return fail(JNX_ERR_UNSUPPORTED, "backbone: d_model %d not in {256..4096}", d);
    const int qkvw = (bb->n_heads + 2 * bb->n_kv_heads) * bb->head_dim;
    jnx_status st;
    if ((st = gemm_check(1, qkvw, d)) || (st = gemm_check(1, d, bb->n_heads * bb->head_dim)) ||
        (st = gemm_check(1, 2 * bb->d_ff, d)) || (st = gemm_check(1, d, bb->d_ff)))
        return st;
    if (bb->glu != JNX_GLU_SWIGLU && bb->glu != JNX_GLU_GEGLU_TANH)
        return fail(JNX_ERR_INVALID_ARG, "backbone: unknown glu %d", bb->glu);
    if (bb->lora_rank != 0 && bb->lora_rank != kLoraRank)
        return fail(JNX_ERR_UNSUPPORTED, "backbone: LoRA rank %d (built for %d)", bb->lora_rank,
                    kLoraRank);
    if (bb->lora_rank && (bb->n_tenants <= 0 || d % 64 || (bb->n_heads * bb->head_dim) % 64))
        return fail(JNX_ERR_INVALID_ARG, "backbone: LoRA needs n_tenants > 0 and widths %% 64");
    for (int l = 0; l < bb->n_layers; ++l) {
        const jnx_layer& L = bb->layers[l];
        if (!L.attn_norm || !L.w_qkv || !L.w_o || !L.ffn_norm || !L.w_gu || !L.w_down)
            return fail(JNX_ERR_INVALID_ARG, "backbone: layer %d has a null weight", l);
        if (bb->lora_rank && (!L.lora_a_q || !L.lora_b_q || !L.lora_a_k || !L.lora_b_k ||
                              !L.lora_a_v || !L.lora_b_v || !L.lora_a_o || !L.lora_b_o))
            return fail(JNX_ERR_INVALID_ARG, "backbone: layer %d has a null LoRA adapter", l);
    }
    return JNX_OK;
}

jnx_status check_group(const jnx_group* g) {
    if (!g) return fail(JNX_ERR_INVALID_ARG, "group: null");
    if (g->n_samples < 0 || g->n_tokens < 0 || g->n_slots < 0 || g->max_seqlen < 0)
        return fail(JNX_ERR_INVALID_ARG, "group: negative count");
    if (g->n_samples > 0 && (!g->cu_seqlens || !g->sample_slot || !g->sample_target ||
                             !g->h_cu_seqlens))
        return fail(JNX_ERR_INVALID_ARG, "group: null sample array");
    if (g->n_tokens > 0 && (!g->gather_src || !g->pos_ids))
        return fail(JNX_ERR_INVALID_ARG, "group: null token array");
    if (g->n_slots > 0 && (!g->seg_offsets || !g->h_seg_offsets || !g->h_slot_tenant))
        return fail(JNX_ERR_INVALID_ARG, "group: null slot array");
    if (g->max_seqlen > kMaxRopePos)
        return fail(JNX_ERR_UNSUPPORTED, "group: sample longer than %d tokens", kMaxRopePos);
    if (g->n_attn_items < 0 || (g->n_attn_items > 0 && !g->attn_items) ||
        (reinterpret_cast<uintptr_t>(g->attn_items) & 7))
        return fail(JNX_ERR_INVALID_ARG, "group: bad attention work list");
    return JNX_OK;
}

// The work list the attention launches take: the group's own device copy
// when it has one (checked against the plan), else `upload` (uploaded here
// from host memory, which a capturing stream refuses).
jnx_status attn_items_for(const jnx_group* g, int2* upload, cudaStream_t s, const char* what,
                          const int2*& items, int& n_items) {
    jnx_status st;
    std::vector<int2> sorted;
    if ((st = build_attn_items(g, sorted))) return st;
    n_items = (int)sorted.size();
    if (g->attn_items) {
        if (g->n_attn_items != n_items)
            return fail(JNX_ERR_INVALID_ARG, "%s: the group's work list has %d items, its plan %d",
                        what, g->n_attn_items, n_items);
        items = reinterpret_cast<const int2*>(g->attn_items);
        return JNX_OK;
    }
    if ((st = refuse_capture(s, what))) return st;
    if (n_items && cudaMemcpyAsync(upload, sorted.data(), sorted.size() * sizeof(int2),
                                   cudaMemcpyHostToDevice, s) != cudaSuccess)
        return fail(JNX_ERR_CUDA, "%s: attention items: %s", what,
                    cudaGetErrorString(cudaGetLastError()));
    items = upload;
    return JNX_OK;
}

// Attention work items (sample, 128-row tile), most expensive first, so
// that a persistent kernel's round-robin over them ends with the cheap ones
// (longest-processing-time-first balance across SMs).  The same list serves
// every layer, the forward and the backward: the samples do not change.
jnx_status build_attn_items(const jnx_group* g, std::vector<int2>& sorted) {
    std::vector<int2> items;
    std::vector<int> cost;
    for (int i = 0; i < g->n_samples; ++i) {
        const int L = g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i];
        for (int q0 = 0; q0 < L; q0 += 128) {
            items.push_back(make_int2(i, q0 / 128));
            cost.push_back((L + 63) / 64);  // 64-row tiles the item's loop walks
        }
    }
    std::vector<int> order(items.size());
    for (size_t i = 0; i < order.size(); ++i) order[i] = (int)i;
    std::stable_sort(order.begin(), order.end(), [&](int a, int b) { return cost[a] > cost[b]; });
    sorted.resize(items.size());
    for (size_t i = 0; i < order.size(); ++i) sorted[i] = items[order[i]];
    if (sorted.size() > (size_t)g->n_tokens + g->n_tokens / 128 + 1)
        return fail(JNX_ERR_INVALID_ARG, "attention items: sample lengths exceed n_tokens");
    return JNX_OK;
}

}  // namespace jnx

extern "C" size_t jnx_backbone_workspace_bytes(const jnx_backbone* bb, int32_t n_tokens) {
    if (!bb || n_tokens < 0) return 0;
    return carve_backbone(bb, n_tokens, nullptr).bytes;
}

// The forward; with `saved`, also keeps each block's fp32 residual input
// and the final residual ([n_layers + 1, N, d]) for the adapter backward.
static jnx_status backbone_forward(const jnx_backbone* bb, const jnx_group* g,
                                   const uint16_t* vision, int64_t n_vision_rows,
                                   const int32_t* text_ids, int64_t n_text, float* pooled,
                                   uint16_t* hidden, float* saved, void* workspace, size_t ws_bytes,
                                   void* stream) {
    jnx_status st;
    if ((st = check_backbone(bb)) || (st = check_group(g))) return st;
    if (!workspace) return fail(JNX_ERR_INVALID_ARG, "backbone: null workspace");
    const int N = g->n_tokens, d = bb->d_model, H = bb->n_heads, Hkv = bb->n_kv_heads,
              hd = bb->head_dim, F = bb->d_ff;
    BackboneWs w = carve_backbone(bb, N, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "backbone: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    if (N == 0) return JNX_OK;
    const bool lora = bb->lora_rank != 0;
    for (int i = 0; lora && i < g->n_slots; ++i)
        if (g->h_slot_tenant[i] < 0 || g->h_slot_tenant[i] >= bb->n_tenants)
            return fail(JNX_ERR_INVALID_ARG, "backbone: tenant %d has no LoRA adapter",
                        g->h_slot_tenant[i]);
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int2* items = nullptr;
    int n_items = 0;
    if ((st = attn_items_for(g, w.attn_items, s, "backbone", items, n_items))) return st;
    const int qkvw = (H + 2 * Hkv) * hd;

    const double Nd = (double)N * d;
    {
        TraceScope ts(JNX_K_PACK, Nd * 6.0, s);
        if ((st = pack_launch(g, vision, n_vision_rows, text_ids, n_text, bb->text_table,
                              bb->vocab, d, w.x, w.status, s)))
            return st;
    }
    {
        TraceScope ts(JNX_K_ROPE_TABLE, (double)g->max_seqlen * hd * 4.0, s);
        if ((st = rope_table_launch(w.rope, g->max_seqlen, hd, bb->rope_theta, s))) return st;
    }
    // LoRA: one segment per group tenant (its contiguous packed rows)
    std::vector<int> seg_r0, seg_r1;
    LoraSpec lq{}, lo{};
    if (lora) {
        if (g->n_slots > kLoraMaxSlots)
            return fail(JNX_ERR_UNSUPPORTED, "backbone: LoRA groups hold at most %d tenants",
                        kLoraMaxSlots);
        for (int i = 0; i < g->n_slots; ++i) {
            seg_r0.push_back(g->h_cu_seqlens[g->h_seg_offsets[i]]);
            seg_r1.push_back(g->h_cu_seqlens[g->h_seg_offsets[i + 1]]);
        }
        lq.t = w.t_qkv;
        lq.ldt = 3 * kLoraRank;
        lq.n_parts = 3;
        lq.cols[0] = H * hd;
        lq.cols[1] = Hkv * hd;
        lq.cols[2] = Hkv * hd;
        lo.t = w.t_o;
        lo.ldt = kLoraRank;
        lo.n_parts = 1;
        lo.cols[0] = d;
        for (LoraSpec* ls : {&lq, &lo}) {
            ls->n_tenants = bb->n_tenants;
            ls->n_seg = g->n_slots;
            ls->seg_r0 = seg_r0.data();
            ls->seg_r1 = seg_r1.data();
            ls->seg_tenant = g->h_slot_tenant;
        }
    }
    // within-sample attention FLOPs: QK^T and PV over each sample's own tokens
    double attn_flops = 0.0;
    for (int i = 0; i < g->n_samples; ++i) {
        const double L = g->h_cu_seqlens[i + 1] - g->h_cu_seqlens[i];
        attn_flops += 4.0 * L * L * H * hd;
    }

    // Fold an RMSNorm into the residual GEMM before it only where that GEMM's
    // K loop is long enough to hide the extra epilogue work (writing y and
    // the sums of squares).  Measured on GB300: at K = 4096 (7B-class O
    // projection) the fold saves ~0.12 ms per launch against k_rmsnorm, at
    // K = 2048 (2B-class O projection) it costs ~0.2 ms more.
    const bool fold_ffn = H * hd >= 4096;  // pre-FFN norm, after the O projection
    const bool fold_attn = F >= 4096;      // pre-attention norm, after the down projection
    auto save = [&](int l) -> jnx_status {
        if (!saved) return JNX_OK;
        return cudaMemcpyAsync(saved + (size_t)l * N * d, w.x, (size_t)N * d * sizeof(float),
                               cudaMemcpyDeviceToDevice, s) == cudaSuccess
                   ? JNX_OK
                   : cuda_status("backbone: saving a residual");
    };
    for (int l = 0; l < bb->n_layers; ++l) {
        const jnx_layer& L = bb->layers[l];
        if ((st = save(l))) return st;
        // attention sub-block.  A folded RMSNorm: the residual GEMM before it
        // (or, for the first block, rms_prep) writes y = bf16(x * gamma) and
        // the row's sums of x^2; the GEMM after it reads y and scales each
        // output row by rsqrt(mean(x^2) + eps).  Unfolded: k_rmsnorm.
        if (l == 0 && fold_attn) {
            TraceScope ts(JNX_K_RMSNORM, Nd * 6.0, s);
            if ((st = rms_prep_launch(w.x, L.attn_norm, N, d, w.nrm, w.ss, s))) return st;
        } else if (!fold_attn) {
            TraceScope ts(JNX_K_RMSNORM, Nd * 6.0, s);
            if ((st = rmsnorm_launch(w.x, L.attn_norm, bb->eps, N, d, w.nrm, s))) return st;
        }
        auto fold_in = [&](GemmParams& q) {
            q.ss_in = w.ss;
            q.ss_parts = d / 128;
            q.ss_cols = d;
            q.ss_eps = bb->eps;
        };
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
        if (fold_attn) fold_in(p);
        if (lora) {
            {
                TraceScope ts(JNX_K_LORA, 2.0 * N * d * 3 * kLoraRank, s);
                const uint16_t* a3[3] = {L.lora_a_q, L.lora_a_k, L.lora_a_v};
                if ((st = lora_down_launch(g, w.nrm, d, d, 3, a3, w.t_qkv, 3 * kLoraRank, s)))
                    return st;
            }
            lq.b[0] = L.lora_b_q;
            lq.b[1] = L.lora_b_k;
            lq.b[2] = L.lora_b_v;
            TraceScope ts(JNX_K_GEMM_QKV, 2.0 * N * qkvw * d, s);
            if ((st = gemm_launch_lora(w.nrm, d, L.w_qkv, d, p, lq, s))) return st;
        } else {
            TraceScope ts(JNX_K_GEMM_QKV, 2.0 * N * qkvw * d, s);
            if ((st = gemm_launch(w.nrm, d, L.w_qkv, d, p, s))) return st;
        }
        {
            TraceScope ts(JNX_K_ATTN, attn_flops, s);
            if ((st = attention_launch(w.qkv, qkvw, N, H, Hkv, hd, g->cu_seqlens, g->n_samples,
                                       g->max_seqlen, items, n_items, w.att, H * hd,
                                       nullptr, w.status, s)))
                return st;
        }
        p = GemmParams{};
        p.M = N;
        p.N = d;
        p.K = H * hd;
        p.epi = EPI_RESID;
        p.resid = w.x;
        p.ldr = d;
        p.status = w.status;
        if (fold_ffn) {  // the pre-FFN norm's first half
            p.norm_gamma = L.ffn_norm;
            p.norm_out = w.nrm;
            p.ss_out = w.ss;
        }
        if (lora) {
            {
                TraceScope ts(JNX_K_LORA, 2.0 * N * H * hd * kLoraRank, s);
                const uint16_t* a1[1] = {L.lora_a_o};
                if ((st = lora_down_launch(g, w.att, H * hd, H * hd, 1, a1, w.t_o, kLoraRank, s)))
                    return st;
            }
            lo.b[0] = L.lora_b_o;
            TraceScope ts(JNX_K_GEMM_O, 2.0 * N * d * H * hd, s);
            if ((st = gemm_launch_lora(w.att, H * hd, L.w_o, H * hd, p, lo, s))) return st;
        } else {
            TraceScope ts(JNX_K_GEMM_O, 2.0 * N * d * H * hd, s);
            if ((st = gemm_launch(w.att, H * hd, L.w_o, H * hd, p, s))) return st;
        }
        // feed-forward sub-block
        if (!fold_ffn) {
            TraceScope ts(JNX_K_RMSNORM, Nd * 6.0, s);
            if ((st = rmsnorm_launch(w.x, L.ffn_norm, bb->eps, N, d, w.nrm, s))) return st;
        }
        p = GemmParams{};
        p.M = N;
        p.N = 2 * F;
        p.K = d;
        p.epi = EPI_GLU;
        p.out = w.u;
        p.ldo = F;
        p.act = bb->glu;
        p.status = w.status;
        if (fold_ffn) fold_in(p);
        {
            TraceScope ts(JNX_K_GEMM_GU, 2.0 * N * 2.0 * F * d, s);
            if ((st = gemm_launch(w.nrm, d, L.w_gu, d, p, s))) return st;
        }
        p = GemmParams{};
        p.M = N;
        p.N = d;
        p.K = F;
        p.epi = EPI_RESID;
        p.resid = w.x;
        p.ldr = d;
        p.status = w.status;
        if (fold_attn && l + 1 < bb->n_layers) {  // the next block's pre-attention norm
            p.norm_gamma = bb->layers[l + 1].attn_norm;
            p.norm_out = w.nrm;
            p.ss_out = w.ss;
        }
        {
            TraceScope ts(JNX_K_GEMM_DOWN, 2.0 * N * d * F, s);
            if ((st = gemm_launch(w.u, F, L.w_down, F, p, s))) return st;
        }
    }
    if ((st = save(bb->n_layers))) return st;
    TraceScope ts(JNX_K_POOL, Nd * 4.0 + (hidden ? Nd * 2.0 : 0.0) +
                                  (pooled ? (double)g->n_samples * d * 4.0 : 0.0), s);
    return final_pool_launch(w.x, bb->final_norm, bb->eps, g->cu_seqlens, g->n_samples, d, pooled,
                             hidden, s);
}

extern "C" int32_t jnx_group_attn_items(const jnx_group* g, int32_t* out, int32_t cap) {
    clear_error();
    if (!g || g->n_samples < 0 || g->n_tokens < 0 || (g->n_samples > 0 && !g->h_cu_seqlens)) {
        fail(JNX_ERR_INVALID_ARG, "group attention items: bad group");
        return JNX_ERR_INVALID_ARG;
    }
    std::vector<int2> sorted;
    jnx_status st = build_attn_items(g, sorted);
    if (st) return st;
    const int32_t n = (int32_t)sorted.size();
    if (!out || cap < n) return n;
    for (int32_t i = 0; i < n; ++i) {
        out[2 * i] = sorted[i].x;
        out[2 * i + 1] = sorted[i].y;
    }
    return n;
}

extern "C" jnx_status jnx_backbone_forward(const jnx_backbone* bb, const jnx_group* g,
                                           const uint16_t* vision, int64_t n_vision_rows,
                                           const int32_t* text_ids, int64_t n_text, float* pooled,
                                           uint16_t* hidden, void* workspace, size_t ws_bytes,
                                           void* stream) {
    clear_error();
    return backbone_forward(bb, g, vision, n_vision_rows, text_ids, n_text, pooled, hidden,
                            nullptr, workspace, ws_bytes, stream);
}

extern "C" size_t jnx_backbone_saved_bytes(const jnx_backbone* bb, int32_t n_tokens) {
    if (!bb || n_tokens < 0 || bb->n_layers < 0) return 0;
    return (size_t)(bb->n_layers + 1) * (size_t)n_tokens * (size_t)bb->d_model * sizeof(float);
}

extern "C" jnx_status jnx_backbone_forward_train(const jnx_backbone* bb, const jnx_group* g,
                                                 const uint16_t* vision, int64_t n_vision_rows,
                                                 const int32_t* text_ids, int64_t n_text,
                                                 float* pooled, uint16_t* hidden, float* saved,
                                                 void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    if (!saved) return fail(JNX_ERR_INVALID_ARG, "backbone: null saved-activation buffer");
    return backbone_forward(bb, g, vision, n_vision_rows, text_ids, n_text, pooled, hidden, saved,
                            workspace, ws_bytes, stream);
}

// ---------------------------------------------------------------------------
// heads
// ---------------------------------------------------------------------------
namespace {

struct HeadsWs {
    int* status;
    HeadScratch sc;
    size_t bytes;
};

struct HeadDims {
    int ld_h = 8, ld_y = 8, ldkv = 256, nq = 4, d_in = 128;
    bool any_mlp = false, any_x = false;
};

int head_hid(const jnx_head& h) {
    return h.kind == JNX_HEAD_MLP ? h.d_hidden : h.n_queries * h.q_dim;
}

HeadDims head_dims(const jnx_head* heads, const jnx_group* g) {
    HeadDims d;
    for (int i = 0; i < g->n_slots; ++i) {
        const jnx_head& h = heads[g->h_slot_tenant[i]];
        d.ld_h = std::max(d.ld_h, head_hid(h));
        d.ld_y = std::max(d.ld_y, h.width);
        if (h.kind == JNX_HEAD_XATTN) {
            d.any_x = true;
            d.ldkv = std::max(d.ldkv, h.q_dim);
            d.nq = h.n_queries;
            d.d_in = std::max(d.d_in, h.d_in);
        } else {
            d.any_mlp = true;
        }
    }
    d.ld_h = (d.ld_h + 7) / 8 * 8;
    d.ld_y = (d.ld_y + 7) / 8 * 8;
    return d;
}

HeadsWs carve_heads(const jnx_head* heads, const jnx_group* g, void* base) {
    uint8_t* p = static_cast<uint8_t*>(base);
    HeadsWs w{};
    size_t off = 0;
    auto take = [&](size_t bytes) {
        uint8_t* r = p ? p + off : nullptr;
        off += up(bytes);
        return reinterpret_cast<float*>(r);
    };
    const HeadDims hd = head_dims(heads, g);
    const size_t S = (size_t)std::max(g->n_samples, 1), N = (size_t)std::max(g->n_tokens, 1);
    w.status = reinterpret_cast<int*>(take(kStatusBytes));
    w.sc.ld_h = hd.ld_h;
    w.sc.ld_y = hd.ld_y;
    w.sc.z = take(S * hd.ld_h * 4);
    w.sc.h = take(S * hd.ld_h * 4);
    w.sc.dh = take(S * hd.ld_h * 4);
    w.sc.y = take(S * hd.ld_y * 4);
    w.sc.dy = take(S * hd.ld_y * 4);
    w.sc.ldkv = hd.ldkv;
    if (hd.any_x) {
        w.sc.kbuf = take(N * hd.ldkv * 4);
        w.sc.vbuf = take(N * hd.ldkv * 4);
        w.sc.dk = take(N * hd.ldkv * 4);
        w.sc.dv = take(N * hd.ldkv * 4);
        w.sc.P = take(N * hd.nq * 4);
        w.sc.dS = take(N * hd.nq * 4);
        w.sc.dQs = take(S * hd.ld_h * 4);
        w.sc.dkv_bf = reinterpret_cast<uint16_t*>(take(N * 2 * hd.ldkv * 2));
        w.sc.Gs = take(S * 32 * hd.d_in * 4);
        w.sc.Hs = take(S * 32 * hd.d_in * 4);
    }
    w.bytes = off;
    return w;
}

jnx_status check_heads(const jnx_head* heads, int32_t n_tenants, const jnx_group* g,
                       bool need_grads, const jnx_head_grads* grads, const float* pooled,
                       const uint16_t* hidden) {
    jnx_status st;
    if ((st = check_group(g))) return st;
    if (!heads && g->n_slots > 0) return fail(JNX_ERR_INVALID_ARG, "heads: null head table");
    int nq = -1;
    for (int i = 0; i < g->n_slots; ++i) {
        const int t = g->h_slot_tenant[i];
        if (t < 0 || t >= n_tenants)
            return fail(JNX_ERR_INVALID_ARG, "heads: group slot %d tenant %d out of range", i, t);
        const jnx_head& h = heads[t];
        if (h.width <= 0 || h.d_in <= 0 || h.d_in % 64)
            return fail(JNX_ERR_UNSUPPORTED, "heads: tenant %d needs width > 0, d_in %% 64 == 0", t);
        if (h.d_in != heads[g->h_slot_tenant[0]].d_in)
            return fail(JNX_ERR_UNSUPPORTED,
                        "heads: the heads of one group read the same features (one d_in)");
        if (h.kind == JNX_HEAD_MLP) {
            if (h.d_hidden <= 0 || h.d_hidden % 8)
                return fail(JNX_ERR_UNSUPPORTED, "heads: tenant %d d_hidden %% 8 != 0", t);
            if (!h.w1 || !h.b1 || !h.w2 || !h.b2)
                return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d null parameter", t);
            if (!pooled) return fail(JNX_ERR_INVALID_ARG, "heads: MLP heads need pooled features");
            if (need_grads && (!grads[t].w1 || !grads[t].b1 || !grads[t].w2 || !grads[t].b2))
                return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d null gradient buffer", t);
        } else if (h.kind == JNX_HEAD_XATTN) {
            if (h.n_queries <= 0 || h.n_queries > 32 || h.n_queries % 4 || h.q_dim % 256 ||
                h.q_dim > 512 || h.q_dim <= 0)
                return fail(JNX_ERR_UNSUPPORTED,
                            "heads: tenant %d query head needs n_queries in {4,8,..,32} and "
                            "q_dim in {256, 512}", t);
            if (nq >= 0 && nq != h.n_queries)
                return fail(JNX_ERR_UNSUPPORTED, "heads: query heads of one group differ in n_queries");
            nq = h.n_queries;
            if (!h.q || !h.wk || !h.wv || !h.wout || !h.bout)
                return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d null parameter", t);
            if (reinterpret_cast<uintptr_t>(h.q) & 15)
                return fail(JNX_ERR_INVALID_ARG,
                            "heads: tenant %d learned queries must be 16-byte aligned", t);
            if (!hidden) return fail(JNX_ERR_INVALID_ARG, "heads: query heads need hidden rows");
            if (h.d_in % 128)
                return fail(JNX_ERR_UNSUPPORTED, "heads: query heads need d_in %% 128 == 0");
            if (need_grads && (!grads[t].q || !grads[t].wk || !grads[t].wv || !grads[t].wout ||
                               !grads[t].bout))
                return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d null gradient buffer", t);
        } else {
            return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d unknown head kind %d", t, h.kind);
        }
        // weight rows are read, and the output layer's gradients written, with
        // 16-byte accesses
        auto a16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; };
        const uint16_t* w_out = h.kind == JNX_HEAD_MLP ? h.w2 : h.wout;
        if (!a16(w_out) || (h.kind == JNX_HEAD_MLP && !a16(h.w1)))
            return fail(JNX_ERR_INVALID_ARG, "heads: tenant %d weights must be 16-byte aligned", t);
        if (need_grads) {
            const float* gw = h.kind == JNX_HEAD_MLP ? grads[t].w2 : grads[t].wout;
            if (!a16(gw) || (h.kind == JNX_HEAD_XATTN && (!a16(grads[t].wk) || !a16(grads[t].wv))))
                return fail(JNX_ERR_INVALID_ARG,
                            "heads: tenant %d gradient buffers must be 16-byte aligned", t);
        }
        const int s0 = g->h_seg_offsets[i], s1 = g->h_seg_offsets[i + 1];
        if (s0 < 0 || s1 <= s0 || s1 > g->n_samples)
            return fail(JNX_ERR_INVALID_ARG, "heads: bad segment of group slot %d", i);
    }
    return JNX_OK;
}

// Fill the per-slot table for group slots [g0, g0 + n) and describe the batch.
HeadBatch fill_table(HeadTable& tab, const jnx_head* heads, const jnx_head_grads* grads,
                     const jnx_group* g, int g0, int n, bool accum = false) {
    HeadBatch b{};
    b.g0 = g0;
    b.n = n;
    b.sample0 = g->h_seg_offsets[g0];
    b.sample1 = g->h_seg_offsets[g0 + n];
    for (int i = 0; i < n; ++i) {
        const int t = g->h_slot_tenant[g0 + i];
        const jnx_head& h = heads[t];
        HeadSlot& hs = tab.slot[i];
        hs = HeadSlot{};
        hs.accum = accum ? 1 : 0;
        hs.kind = h.kind;
        hs.tenant = t;
        hs.s0 = g->h_seg_offsets[g0 + i];
        hs.s1 = g->h_seg_offsets[g0 + i + 1];
        hs.r0 = g->h_cu_seqlens[hs.s0];
        hs.r1 = g->h_cu_seqlens[hs.s1];
        hs.d_in = h.d_in;
        hs.hid = head_hid(h);
        hs.width = h.width;
        if (h.kind == JNX_HEAD_MLP) {
            hs.w1 = h.w1;
            hs.b1 = h.b1;
            hs.w2 = h.w2;
            hs.b2 = h.b2;
            if (grads) {
                hs.g_w1 = grads[t].w1;
                hs.g_b1 = grads[t].b1;
                hs.g_w2 = grads[t].w2;
                hs.g_b2 = grads[t].b2;
            }
            b.any_mlp = true;
            b.max_mlp_hid = std::max(b.max_mlp_hid, hs.hid);
        } else {
            hs.nq = h.n_queries;
            hs.dq = h.q_dim;
            hs.w2 = h.wout;
            hs.b2 = h.bout;
            hs.q = h.q;
            hs.wk = h.wk;
            hs.wv = h.wv;
            if (grads) {
                hs.g_w2 = grads[t].wout;
                hs.g_b2 = grads[t].bout;
                hs.g_q = grads[t].q;
                hs.g_wk = grads[t].wk;
                hs.g_wv = grads[t].wv;
            }
            b.any_xattn = true;
            b.max_nq = std::max(b.max_nq, hs.nq);
            b.max_dq = std::max(b.max_dq, hs.dq);
        }
        b.max_hid = std::max(b.max_hid, hs.hid);
        b.max_width = std::max(b.max_width, hs.width);
        b.max_ns = std::max(b.max_ns, hs.s1 - hs.s0);
    }
    return b;
}

double heads_flops(const HeadTable& tab, int n, bool backward) {
    double fl = 0.0;
    for (int i = 0; i < n; ++i) {
        const HeadSlot& h = tab.slot[i];
        const double ns = h.s1 - h.s0, nr = h.r1 - h.r0;
        if (h.kind == JNX_HEAD_MLP) {
            fl += 2.0 * ns * ((double)h.d_in * h.hid + (backward ? 2.0 : 1.0) * h.hid * h.width);
        } else {
            const double kv = 2.0 * nr * h.d_in * 2.0 * h.dq;
            const double att = 4.0 * h.nq * h.dq * nr;
            const double out = 2.0 * ns * h.hid * h.width;
            fl += backward ? (kv + 2.0 * att + 2.0 * out) : (kv + att + out);
        }
    }
    return fl;
}

}  // namespace

extern "C" size_t jnx_heads_workspace_bytes(const jnx_head* heads, int32_t n_tenants,
                                            const jnx_group* g) {
    if (!g || (g->n_slots > 0 && (!heads || !g->h_slot_tenant))) return 0;
    for (int i = 0; i < g->n_slots; ++i)
        if (g->h_slot_tenant[i] < 0 || g->h_slot_tenant[i] >= n_tenants) return 0;
    return carve_heads(heads, g, nullptr).bytes;
}

extern "C" jnx_status jnx_heads_forward(const jnx_head* heads, int32_t n_tenants,
                                        const jnx_group* g, const float* pooled,
                                        const uint16_t* hidden, const float* targets, float* preds,
                                        float* loss, void* workspace, size_t ws_bytes,
                                        void* stream) {
    clear_error();
    jnx_status st;
    if ((st = check_heads(heads, n_tenants, g, false, nullptr, pooled, hidden))) return st;
    if (g->n_slots == 0) return JNX_OK;
    if (!preds || !workspace || (!targets) != (!loss))
        return fail(JNX_ERR_INVALID_ARG, "heads forward: null buffer");
    HeadsWs w = carve_heads(heads, g, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "heads: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    if ((st = heads_set_smem())) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int d = heads[g->h_slot_tenant[0]].d_in;
    HeadTable tab;
    for (int g0 = 0; g0 < g->n_slots; g0 += kMaxSlots) {
        const int n = std::min(kMaxSlots, g->n_slots - g0);
        HeadBatch b = fill_table(tab, heads, nullptr, g, g0, n);
        TraceScope ts(JNX_K_HEADS_FWD, heads_flops(tab, n, false), s);
        for (int i = 0; i < n && b.any_xattn; ++i) {
            const HeadSlot& hs = tab.slot[i];
            if (hs.kind != JNX_HEAD_XATTN || hs.r1 == hs.r0) continue;
            for (int which = 0; which < 2; ++which) {
                GemmParams p{};
                p.M = hs.r1 - hs.r0;
                p.N = hs.dq;
                p.K = d;
                p.epi = EPI_F32;
                p.out = (which ? w.sc.vbuf : w.sc.kbuf) + (size_t)hs.r0 * w.sc.ldkv;
                p.ldo = w.sc.ldkv;
                p.status = w.status;
                if ((st = gemm_launch(hidden + (size_t)hs.r0 * d, d, which ? hs.wv : hs.wk, d, p,
                                      s)))
                    return st;
            }
        }
        if ((st = heads_forward_launch(tab, b, w.sc, pooled, d, g->cu_seqlens, g->sample_slot,
                                       g->sample_target, targets, preds, loss, s)))
            return st;
    }
    return JNX_OK;
}

static jnx_status heads_backward(const jnx_head* heads, int32_t n_tenants, const jnx_group* g,
                                 const float* pooled, const uint16_t* hidden,
                                 const jnx_head_grads* grads, void* workspace, size_t ws_bytes,
                                 void* stream, bool accum, bool kv_grads = false) {
    jnx_status st;
    if (!grads && g && g->n_slots > 0)
        return fail(JNX_ERR_INVALID_ARG, "heads backward: null grads");
    if ((st = check_heads(heads, n_tenants, g, true, grads, pooled, hidden))) return st;
    if (g->n_slots == 0) return JNX_OK;
    if (!workspace) return fail(JNX_ERR_INVALID_ARG, "heads backward: null workspace");
    HeadsWs w = carve_heads(heads, g, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "heads: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    if ((st = heads_set_smem())) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int d = heads[g->h_slot_tenant[0]].d_in;
    HeadTable tab;
    for (int g0 = 0; g0 < g->n_slots; g0 += kMaxSlots) {
        const int n = std::min(kMaxSlots, g->n_slots - g0);
        HeadBatch b = fill_table(tab, heads, grads, g, g0, n, accum);
        TraceScope ts(JNX_K_HEADS_BWD, heads_flops(tab, n, true), s);
        if ((st = heads_backward_launch(tab, b, w.sc, pooled, d, hidden, g->cu_seqlens,
                                        g->sample_slot, kv_grads, s)))
            return st;
    }
    return JNX_OK;
}

extern "C" jnx_status jnx_heads_backward(const jnx_head* heads, int32_t n_tenants,
                                         const jnx_group* g, const float* pooled,
                                         const uint16_t* hidden, const float* targets,
                                         const jnx_head_grads* grads, void* workspace,
                                         size_t ws_bytes, void* stream) {
    clear_error();
    (void)targets;  // the loss gradient dy was kept by the forward
    return heads_backward(heads, n_tenants, g, pooled, hidden, grads, workspace, ws_bytes, stream,
                          false);
}

extern "C" jnx_status jnx_heads_backward_accumulate(const jnx_head* heads, int32_t n_tenants,
                                                    const jnx_group* g, const float* pooled,
                                                    const uint16_t* hidden, const float* targets,
                                                    const jnx_head_grads* grads, void* workspace,
                                                    size_t ws_bytes, void* stream) {
    clear_error();
    (void)targets;
    return heads_backward(heads, n_tenants, g, pooled, hidden, grads, workspace, ws_bytes, stream,
                          true);
}

// dloss_t/d(final normed row) of every token row, after the heads backward
// (which leaves dz of the MLP heads and dk, dv of the query heads in the
// workspace): an MLP sample's rows each get (dz W1) / L; a query-head row
// gets dk W_k + dv W_v.
static jnx_status heads_feature_grad(const jnx_head* heads, const jnx_group* g, float* d_hidden,
                                     void* workspace, cudaStream_t s) {
    if (g->n_slots > kSegMaxSlots)
        return fail(JNX_ERR_UNSUPPORTED, "heads feature gradient: at most %d tenants", kSegMaxSlots);
    HeadsWs w = carve_heads(heads, g, workspace);
    const int d = heads[g->h_slot_tenant[0]].d_in, N = g->n_tokens;
    static thread_local MlpFeatTable mt;
    mt = MlpFeatTable{};
    bool any_mlp = false, any_x = false;
    for (int i = 0; i < g->n_slots; ++i) {
        const jnx_head& h = heads[g->h_slot_tenant[i]];
        if (h.kind == JNX_HEAD_MLP) {
            mt.w1[i] = h.w1;
            mt.hid[i] = h.d_hidden;
            any_mlp = true;
        } else {
            any_x = true;
        }
    }
    jnx_status st;
    TraceScope ts(JNX_K_HEADS_BWD, 0.0, s);
    if (any_mlp && (st = mlp_dfeat_launch(w.sc.dh, w.sc.ld_h, g->cu_seqlens, g->sample_slot,
                                          g->n_samples, mt, d, d_hidden, s)))
        return st;
    if (!any_x) return JNX_OK;
    const int ld = w.sc.ldkv;
    if ((st = to_bf16_launch(w.sc.dk, ld, N, ld, w.sc.dkv_bf, 2 * ld, s)) ||
        (st = to_bf16_launch(w.sc.dv, ld, N, ld, w.sc.dkv_bf + ld, 2 * ld, s)))
        return st;
    // one launch per distinct query width; other slots are skipped
    std::vector<int> widths;
    for (int i = 0; i < g->n_slots; ++i) {
        const jnx_head& h = heads[g->h_slot_tenant[i]];
        if (h.kind == JNX_HEAD_XATTN &&
            std::find(widths.begin(), widths.end(), h.q_dim) == widths.end())
            widths.push_back(h.q_dim);
    }
    static thread_local SegUpParts sp;
    for (int dq : widths) {
        sp = SegUpParts{};
        sp.n_parts = 2;
        sp.t[0] = w.sc.dkv_bf;
        sp.t[1] = w.sc.dkv_bf + ld;
        sp.ldt[0] = sp.ldt[1] = 2 * ld;
        sp.k[0] = sp.k[1] = dq;
        for (int i = 0; i < g->n_slots; ++i) {
            const jnx_head& h = heads[g->h_slot_tenant[i]];
            if (h.kind == JNX_HEAD_XATTN && h.q_dim == dq) {
                sp.w[0][i] = h.wk;
                sp.w[1][i] = h.wv;
            }
        }
        if ((st = seg_up_launch(g, sp, d, d_hidden, d, false, s))) return st;
    }
    return JNX_OK;
}

extern "C" jnx_status jnx_heads_backward_input(const jnx_head* heads, int32_t n_tenants,
                                               const jnx_group* g, const float* pooled,
                                               const uint16_t* hidden, const float* targets,
                                               const jnx_head_grads* grads, float* d_hidden,
                                               void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    (void)targets;
    if (!d_hidden && g && g->n_tokens > 0)
        return fail(JNX_ERR_INVALID_ARG, "heads backward: null feature-gradient buffer");
    jnx_status st = heads_backward(heads, n_tenants, g, pooled, hidden, grads, workspace,
                                   ws_bytes, stream, false, true);
    if (st || g->n_slots == 0) return st;
    return heads_feature_grad(heads, g, d_hidden, workspace, static_cast<cudaStream_t>(stream));
}

// The heads backward with every group tenant's AdamW step fused into it
// (App. A "Actor Consumption and Version Consistency": the step of one
// tenant's own optimizer, nothing shared or averaged across tenants).
extern "C" jnx_status jnx_heads_backward_adamw(const jnx_head* heads, int32_t n_tenants,
                                               const jnx_group* g, const float* pooled,
                                               const uint16_t* hidden, const float* targets,
                                               const jnx_head_grads* grads, int32_t accumulate,
                                               jnx_head_opt* opt, const jnx_adamw* hp,
                                               float* d_hidden, void* workspace, size_t ws_bytes,
                                               void* stream) {
    clear_error();
    (void)targets;  // the loss gradient dy was kept by the forward
    if (!opt || !hp) return fail(JNX_ERR_INVALID_ARG, "heads backward adamw: null argument");
    if (!(hp->lr >= 0.f) || !(hp->beta1 >= 0.f && hp->beta1 < 1.f) ||
        !(hp->beta2 >= 0.f && hp->beta2 < 1.f) || !(hp->eps >= 0.f) || !(hp->weight_decay >= 0.f))
        return fail(JNX_ERR_INVALID_ARG, "heads backward adamw: hyperparameter out of range");
    if (accumulate && !grads && g && g->n_slots > 0)
        return fail(JNX_ERR_INVALID_ARG, "heads backward adamw: accumulating needs grads");
    jnx_status st;
    if ((st = check_heads(heads, n_tenants, g, accumulate != 0, grads, pooled, hidden))) return st;
    if (g->n_slots == 0) return JNX_OK;
    if (!workspace) return fail(JNX_ERR_INVALID_ARG, "heads backward adamw: null workspace");
    // every group tenant's optimizer state, checked before anything is written
    auto al = [](const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; };
    for (int i = 0; i < g->n_slots; ++i) {
        const int t = g->h_slot_tenant[i];
        const jnx_head& h = heads[t];
        const jnx_head_opt& o = opt[t];
        const bool mlp = h.kind == JNX_HEAD_MLP;
        const int ks[5] = {mlp ? 0 : 4, mlp ? 1 : 5, mlp ? 2 : 6, mlp ? 3 : 7, mlp ? -1 : 8};
        for (int k : ks) {
            if (k < 0) continue;
            if (!o.master[k] || !o.m[k] || !o.v[k])
                return fail(JNX_ERR_INVALID_ARG,
                            "heads backward adamw: tenant %d: null state for tensor %d", t, k);
        }
        // the weight tensors' state is updated with 16-byte (W1, W2, Wout)
        // or 8-byte (Wk, Wv) accesses
        const int vec[3] = {mlp ? 0 : 7, mlp ? 2 : 5, mlp ? -1 : 6};
        for (int k : vec) {
            if (k < 0) continue;
            const uintptr_t a = (k == 5 || k == 6) ? 8 : 16;
            if (!al(o.master[k], a) || !al(o.m[k], a) || !al(o.v[k], a))
                return fail(JNX_ERR_INVALID_ARG,
                            "heads backward adamw: tenant %d: tensor %d state misaligned", t, k);
        }
        if (!mlp && (!al(h.wk, 4) || !al(h.wv, 4)))
            return fail(JNX_ERR_INVALID_ARG, "heads backward adamw: tenant %d: Wk/Wv misaligned", t);
    }
    HeadsWs w = carve_heads(heads, g, workspace);
    if (ws_bytes < w.bytes)
        return fail(JNX_ERR_WORKSPACE, "heads: workspace %zu < %zu bytes", ws_bytes, w.bytes);
    if ((st = heads_set_smem())) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const int d = heads[g->h_slot_tenant[0]].d_in;
    const AdamHp ahp{hp->lr, hp->beta1, hp->beta2, hp->eps, hp->weight_decay};
    static thread_local HeadTable tab;
    static thread_local HeadOptTable otab;
    {
        TraceScope ts(JNX_K_HEADS_BWD, 0.0, s);
        for (int g0 = 0; g0 < g->n_slots; g0 += kMaxSlots) {
            const int n = std::min(kMaxSlots, g->n_slots - g0);
            HeadBatch b = fill_table(tab, heads, grads, g, g0, n, accumulate != 0);
            if ((st = heads_backward_front_launch(tab, b, w.sc, d, hidden, g->cu_seqlens,
                                                  g->sample_slot, d_hidden != nullptr, s)))
                return st;
        }
    }
    if (d_hidden && (st = heads_feature_grad(heads, g, d_hidden, workspace, s))) return st;
    double fl = 0.0;
    for (int g0 = 0; g0 < g->n_slots; g0 += kMaxSlots) {
        const int n = std::min(kMaxSlots, g->n_slots - g0);
        HeadBatch b = fill_table(tab, heads, grads, g, g0, n, accumulate != 0);
        fl += heads_flops(tab, n, true);
        otab = HeadOptTable{};
        for (int i = 0; i < n; ++i) {
            const int t = g->h_slot_tenant[g0 + i];
            const jnx_head& h = heads[t];
            const jnx_head_opt& o = opt[t];
            HeadOpt& ho = otab.slot[i];
            const uint16_t* p[9] = {h.w1, h.b1, h.w2, h.b2, h.q, h.wk, h.wv, h.wout, h.bout};
            for (int k = 0; k < 9; ++k) {
                ho.master[k] = o.master[k];
                ho.m[k] = o.m[k];
                ho.v[k] = o.v[k];
                ho.p[k] = const_cast<uint16_t*>(p[k]);
            }
            const int step = o.step + 1;
            ho.c1 = (float)(1.0 / (1.0 - std::pow((double)hp->beta1, step)));
            ho.c2 = (float)(1.0 / (1.0 - std::pow((double)hp->beta2, step)));
        }
        TraceScope ts(JNX_K_HEADS_BWD, heads_flops(tab, n, true), s);
        if ((st = heads_backward_step_launch(tab, otab, ahp, b, w.sc, pooled, d, s))) return st;
    }
    for (int i = 0; i < g->n_slots; ++i) {
        jnx_head_opt& o = opt[g->h_slot_tenant[i]];
        ++o.step;
        ++o.version;
    }
    return JNX_OK;
}

// ---------------------------------------------------------------------------
// status and helpers

// ---------------------------------------------------------------------------

extern "C" jnx_status jnx_check_status(void* workspace, void* stream) {
    clear_error();
    if (!workspace) return fail(JNX_ERR_INVALID_ARG, "check_status: null workspace");
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int v = 0;
    if (cudaMemcpyAsync(&v, workspace, sizeof v, cudaMemcpyDeviceToHost, s) != cudaSuccess ||
        cudaMemsetAsync(workspace, 0, sizeof v, s) != cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return fail(JNX_ERR_CUDA, "check_status: %s", cudaGetErrorString(cudaGetLastError()));
    if (v != 0) return fail(v, "a kernel reported status %d", v);
    return JNX_OK;
}

__global__ void k_pack_gate_up(const uint16_t* __restrict__ wg, const uint16_t* __restrict__ wu,
                               int F, int d, uint16_t* __restrict__ out) {
    const int64_t row = blockIdx.x;  // output row in [0, 2F)
    const int blk = (int)(row / 128), r = (int)(row % 128);
    const int src = (blk / 2) * 128 + r;
    const uint16_t* in = (blk & 1) ? wu : wg;
    const uint4* a = reinterpret_cast<const uint4*>(in + (size_t)src * d);
    uint4* b = reinterpret_cast<uint4*>(out + (size_t)row * d);
    for (int c = threadIdx.x; c < d / 8; c += blockDim.x) b[c] = a[c];
}

extern "C" jnx_status jnx_pack_gate_up(const uint16_t* w_gate, const uint16_t* w_up, int32_t F,
                                       int32_t d, uint16_t* out, void* stream) {
    clear_error();
    if (!w_gate || !w_up || !out || F <= 0 || d <= 0 || F % 128 || d % 8)
        return fail(JNX_ERR_INVALID_ARG, "pack_gate_up: need F %% 128 == 0 and d %% 8 == 0");
    k_pack_gate_up<<<2 * F, 128, 0, static_cast<cudaStream_t>(stream)>>>(w_gate, w_up, F, d, out);
    return cuda_status("pack_gate_up");
}

// ---------------------------------------------------------------------------
// stage-level entry points (jnx_ops.h)
// ---------------------------------------------------------------------------

extern "C" jnx_status jnx_op_pack(const jnx_group* g, const uint16_t* vision,
                                  int64_t n_vision_rows, const int32_t* text_ids, int64_t n_text,
                                  const uint16_t* text_table, int32_t vocab, int32_t d, float* x,
                                  int32_t* status, void* stream) {
    clear_error();
    jnx_status st;
    if ((st = check_group(g))) return st;
    return pack_launch(g, vision, n_vision_rows, text_ids, n_text, text_table, vocab, d, x, status,
                       static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_op_rmsnorm(const float* x, const uint16_t* gamma, float eps, int32_t M,
                                     int32_t d, uint16_t* out, void* stream) {
    clear_error();
    if (M < 0 || !x || !gamma || !out) return fail(JNX_ERR_INVALID_ARG, "rmsnorm: bad argument");
    return rmsnorm_launch(x, gamma, eps, M, d, out, static_cast<cudaStream_t>(stream));
}

extern "C" size_t jnx_op_gemm_workspace_bytes(int32_t max_pos, int32_t head_dim) {
    return kStatusBytes + up((size_t)std::max(max_pos, 1) * std::max(head_dim / 2, 1) * 8);
}

extern "C" jnx_status jnx_op_gemm(const uint16_t* A, const uint16_t* W, int32_t M, int32_t N,
                                  int32_t K, int32_t epilogue, void* out, int32_t ldo,
                                  const int32_t* pos, int32_t max_pos, int32_t rope_cols,
                                  int32_t head_dim, float rope_theta, int32_t act,
                                  void* workspace, size_t ws_bytes, void* stream) {
    clear_error();
    if (!A || !W || !out || M < 0) return fail(JNX_ERR_INVALID_ARG, "gemm: null argument");
    if ((epilogue < EPI_BF16 || epilogue > EPI_ROPE) && epilogue != EPI_GLU_SAVE)
        return fail(JNX_ERR_INVALID_ARG, "gemm: unknown epilogue %d", epilogue);
    if ((epilogue == EPI_GLU || epilogue == EPI_GLU_SAVE) && act != JNX_GLU_SWIGLU &&
        act != JNX_GLU_GEGLU_TANH)
        return fail(JNX_ERR_INVALID_ARG, "gemm: unknown activation %d", act);
    {
        // the epilogues write (and the residual one reads) 16-byte vectors
        const int esz = (epilogue == EPI_F32 || epilogue == EPI_RESID) ? 4 : 2;
        const int width = epilogue == EPI_GLU ? N / 2 : N;
        if (ldo < width || ((size_t)ldo * esz) % 16 || reinterpret_cast<uintptr_t>(out) % 16)
            return fail(JNX_ERR_INVALID_ARG, "gemm: out needs 16-byte aligned rows of >= %d", width);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    GemmParams p{};
    p.M = M;
    p.N = N;
    p.K = K;
    p.epi = epilogue;
    p.out = out;
    p.ldo = ldo;
    p.act = act;
    if (epilogue == EPI_RESID) {
        p.resid = static_cast<float*>(out);
        p.ldr = ldo;
    }
    if (epilogue == EPI_ROPE) {
        if (!pos || !workspace || (head_dim != 64 && head_dim != 128 && head_dim != 256) ||
            max_pos <= 0)
            return fail(JNX_ERR_INVALID_ARG, "gemm rope: need pos, workspace, head_dim");
        if (rope_cols < 0 || rope_cols > N || rope_cols % head_dim)
            return fail(JNX_ERR_INVALID_ARG,
                        "gemm rope: rope_cols %d must be a multiple of head_dim %d within N %d",
                        rope_cols, head_dim, N);
        if (ws_bytes < jnx_op_gemm_workspace_bytes(max_pos, head_dim))
            return fail(JNX_ERR_WORKSPACE, "gemm rope: workspace too small");
        float2* tab = reinterpret_cast<float2*>(static_cast<uint8_t*>(workspace) + kStatusBytes);
        jnx_status st = rope_table_launch(tab, max_pos, head_dim, rope_theta, s);
        if (st) return st;
        p.pos = pos;
        p.rope = tab;
        p.rope_ld = max_pos;
        p.rope_cols = rope_cols;
        p.hd = head_dim;
    }
    if (workspace) p.status = static_cast<int*>(workspace);
    TraceScope ts(JNX_K_GEMM, 2.0 * M * N * K, s);
    return gemm_launch(A, K, W, K, p, s);
}

extern "C" jnx_status jnx_op_attention(const uint16_t* qkv, int32_t n_tokens, int32_t n_heads,
                                       int32_t n_kv_heads, int32_t head_dim,
                                       const int32_t* cu_seqlens, int32_t n_samples,
                                       int32_t max_seqlen, uint16_t* out, int32_t* status,
                                       void* stream) {
    clear_error();
    if (!qkv || !out || (n_samples > 0 && !cu_seqlens) || n_tokens < 0)
        return fail(JNX_ERR_INVALID_ARG, "attention: null argument");
    const int ldq = (n_heads + 2 * n_kv_heads) * head_dim;
    TraceScope ts(JNX_K_ATTN, 0.0, static_cast<cudaStream_t>(stream));
    return attention_launch(qkv, ldq, n_tokens, n_heads, n_kv_heads, head_dim, cu_seqlens,
                            n_samples, max_seqlen, nullptr, 0, out, n_heads * head_dim, nullptr,
                            status, static_cast<cudaStream_t>(stream));
}

extern "C" jnx_status jnx_op_final_pool(const float* x, const uint16_t* gamma, float eps,
                                        const int32_t* cu_seqlens, int32_t n_samples, int32_t d,
                                        float* pooled, uint16_t* hidden, void* stream) {
    clear_error();
    if (!x || !gamma || (n_samples > 0 && !cu_seqlens))
        return fail(JNX_ERR_INVALID_ARG, "final_pool: null argument");
    return final_pool_launch(x, gamma, eps, cu_seqlens, n_samples, d, pooled, hidden,
                             static_cast<cudaStream_t>(stream));
}
