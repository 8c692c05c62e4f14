// jnx_heads_adamw: the tenant-private optimizer step of the action heads.
//
// App. A ("Actor Consumption and Version Consistency"): an optimizer
// microbatch belongs to one tenant; only that tenant's optimizer steps and
// only its policy version increments; optimizer states are never shared or
// averaged across tenants.  Here one launch steps every tenant of a group,
// each on its own parameters, gradients and moments.
//
// AdamW with decoupled weight decay, fp32, four parameter elements a thread:
// the kernel streams the gradient, the two moments and the fp32 master once
// and writes the moments, the master and the bf16 parameter the forward
// reads (30 bytes per element; HBM-bound).
#include <cmath>
#include <vector>

#include "../../include/jnx.h"
#include "jnx_dev.cuh"
#include "jnx_trace.h"

namespace jnx {
namespace {

constexpr int kMaxSeg = 96;  // parameter tensors per launch

struct AdamSeg {
    uint16_t* p;       // bf16 parameter (written)
    float* master;     // fp32 master copy
    float* m;
    float* v;
    const float* g;    // fp32 gradient
    long long n;       // elements
    float c1, c2;      // 1 / (1 - beta1^t), 1 / (1 - beta2^t)
};

struct AdamTable {
    AdamSeg seg[kMaxSeg];
};

// Four elements per thread (16-byte loads) where the segment's arrays allow
// it, then a scalar tail.
__global__ void __launch_bounds__(256) k_adamw(const __grid_constant__ AdamTable tab, float lr,
                                               float b1, float b2, float eps, float wd) {
    const AdamSeg& s = tab.seg[blockIdx.y];
    const long long stride = (long long)gridDim.x * 256;
    const long long t0 = (long long)blockIdx.x * 256 + threadIdx.x;
    const bool vec = ((reinterpret_cast<uintptr_t>(s.g) | reinterpret_cast<uintptr_t>(s.m) |
                       reinterpret_cast<uintptr_t>(s.v) | reinterpret_cast<uintptr_t>(s.master)) &
                      15) == 0 &&
                     (reinterpret_cast<uintptr_t>(s.p) & 7) == 0;
    const long long n4 = vec ? s.n / 4 : 0;
    for (long long i = t0; i < n4; i += stride) {
        const float4 g = reinterpret_cast<const float4*>(s.g)[i];
        float4 m = reinterpret_cast<float4*>(s.m)[i];
        float4 v = reinterpret_cast<float4*>(s.v)[i];
        float4 p = reinterpret_cast<float4*>(s.master)[i];
        p.x = adamw_elem(g.x, m.x, v.x, p.x, s.c1, s.c2, lr, b1, b2, eps, wd);
        p.y = adamw_elem(g.y, m.y, v.y, p.y, s.c1, s.c2, lr, b1, b2, eps, wd);
        p.z = adamw_elem(g.z, m.z, v.z, p.z, s.c1, s.c2, lr, b1, b2, eps, wd);
        p.w = adamw_elem(g.w, m.w, v.w, p.w, s.c1, s.c2, lr, b1, b2, eps, wd);
        reinterpret_cast<float4*>(s.m)[i] = m;
        reinterpret_cast<float4*>(s.v)[i] = v;
        reinterpret_cast<float4*>(s.master)[i] = p;
        reinterpret_cast<uint2*>(s.p)[i] = make_uint2(pack_bf2(p.x, p.y), pack_bf2(p.z, p.w));
    }
    for (long long i = 4 * n4 + t0; i < s.n; i += stride) {
        float m = s.m[i], v = s.v[i];
        const float p = adamw_elem(s.g[i], m, v, s.master[i], s.c1, s.c2, lr, b1, b2, eps, wd);
        s.m[i] = m;
        s.v[i] = v;
        s.master[i] = p;
        s.p[i] = f2bf(p);
    }
}

}  // namespace
}  // namespace jnx

using namespace jnx;

static jnx_status check_hp(const jnx_adamw* hp) {
    if (!(hp->lr >= 0.f) || !(hp->beta1 >= 0.f && hp->beta1 < 1.f) ||
        !(hp->beta2 >= 0.f && hp->beta2 < 1.f) || !(hp->eps >= 0.f) || !(hp->weight_decay >= 0.f))
        return fail(JNX_ERR_INVALID_ARG, "adamw: hyperparameter out of range");
    return JNX_OK;
}

static jnx_status launch_segments(const std::vector<AdamSeg>& segs, const jnx_adamw* hp,
                                  cudaStream_t s) {
    for (size_t a = 0; a < segs.size(); a += kMaxSeg) {
        AdamTable tab;
        const int ns = (int)std::min<size_t>(kMaxSeg, segs.size() - a);
        long long mx = 0;
        for (int k = 0; k < ns; ++k) {
            tab.seg[k] = segs[a + k];
            mx = std::max(mx, segs[a + k].n);
        }
        if (mx == 0) continue;
        const int bx = (int)std::min<long long>((mx / 4 + 255) / 256 + 1, 1024);
        k_adamw<<<dim3(bx, ns), 256, 0, s>>>(tab, hp->lr, hp->beta1, hp->beta2, hp->eps,
                                             hp->weight_decay);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return fail(JNX_ERR_CUDA, "adamw: %s", cudaGetErrorString(e));
    }
    return JNX_OK;
}

extern "C" jnx_status jnx_adamw_tensors(const jnx_adam_tensor* tensors, int32_t n_tensors,
                                        const jnx_adamw* hp, void* stream) {
    clear_error();
    if (!hp || n_tensors < 0 || (n_tensors > 0 && !tensors))
        return fail(JNX_ERR_INVALID_ARG, "adamw: null argument");
    jnx_status st;
    if ((st = check_hp(hp))) return st;
    std::vector<AdamSeg> segs;
    double bytes = 0.0;
    for (int i = 0; i < n_tensors; ++i) {
        const jnx_adam_tensor& t = tensors[i];
        if (t.n < 0 || !t.step) return fail(JNX_ERR_INVALID_ARG, "adamw: tensor %d", i);
        if (t.n > 0 && (!t.param || !t.master || !t.m || !t.v || !t.grad))
            return fail(JNX_ERR_INVALID_ARG, "adamw: tensor %d has a null buffer", i);
        const int step = *t.step + 1;
        const float c1 = (float)(1.0 / (1.0 - std::pow((double)hp->beta1, step)));
        const float c2 = (float)(1.0 / (1.0 - std::pow((double)hp->beta2, step)));
        segs.push_back(AdamSeg{t.param, t.master, t.m, t.v, t.grad, t.n, c1, c2});
        bytes += 30.0 * (double)t.n;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    {
        TraceScope ts(JNX_K_ADAMW, bytes, s);
        if ((st = launch_segments(segs, hp, s))) return st;
    }
    for (int i = 0; i < n_tensors; ++i) ++*tensors[i].step;
    return JNX_OK;
}

extern "C" jnx_status jnx_heads_adamw(const jnx_head* heads, const jnx_head_grads* grads,
                                      jnx_head_opt* opt, int32_t n_tenants, const jnx_group* g,
                                      const jnx_adamw* hp, void* stream) {
    clear_error();
    if (!heads || !grads || !opt || !g || !hp || n_tenants < 0)
        return fail(JNX_ERR_INVALID_ARG, "adamw: null argument");
    jnx_status st;
    if ((st = check_hp(hp))) return st;
    if (g->n_slots == 0) return JNX_OK;
    if (!g->h_slot_tenant) return fail(JNX_ERR_INVALID_ARG, "adamw: null slot tenants");

    // Every tensor of every group tenant, checked before anything is written.
    std::vector<AdamSeg> segs;
    double bytes = 0.0;
    for (int i = 0; i < g->n_slots; ++i) {
        const int t = g->h_slot_tenant[i];
        if (t < 0 || t >= n_tenants) return fail(JNX_ERR_INVALID_ARG, "adamw: tenant %d", t);
        const jnx_head& h = heads[t];
        const jnx_head_grads& gr = grads[t];
        const jnx_head_opt& o = opt[t];
        long long n[9] = {0, 0, 0, 0, 0, 0, 0, 0, 0};
        if (h.kind == JNX_HEAD_MLP) {
            n[0] = (long long)h.d_hidden * h.d_in;
            n[1] = h.d_hidden;
            n[2] = (long long)h.width * h.d_hidden;
            n[3] = h.width;
        } else if (h.kind == JNX_HEAD_XATTN) {
            n[4] = (long long)h.n_queries * h.q_dim;
            n[5] = (long long)h.q_dim * h.d_in;
            n[6] = (long long)h.q_dim * h.d_in;
            n[7] = (long long)h.width * h.n_queries * h.q_dim;
            n[8] = h.width;
        } else {
            return fail(JNX_ERR_INVALID_ARG, "adamw: tenant %d: unknown head kind %d", t, h.kind);
        }
        const uint16_t* p[9] = {h.w1, h.b1, h.w2, h.b2, h.q, h.wk, h.wv, h.wout, h.bout};
        const float* gg[9] = {gr.w1, gr.b1, gr.w2, gr.b2, gr.q, gr.wk, gr.wv, gr.wout, gr.bout};
        const int step = o.step + 1;
        const float c1 = (float)(1.0 / (1.0 - std::pow((double)hp->beta1, step)));
        const float c2 = (float)(1.0 / (1.0 - std::pow((double)hp->beta2, step)));
        for (int k = 0; k < 9; ++k) {
            if (n[k] <= 0) continue;
            if (!p[k] || !gg[k] || !o.master[k] || !o.m[k] || !o.v[k])
                return fail(JNX_ERR_INVALID_ARG, "adamw: tenant %d: null state for tensor %d", t,
                            k);
            segs.push_back(AdamSeg{const_cast<uint16_t*>(p[k]), o.master[k], o.m[k], o.v[k],
                                   gg[k], n[k], c1, c2});
            bytes += 30.0 * (double)n[k];
        }
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    {
        TraceScope ts(JNX_K_ADAMW, bytes, s);
        if ((st = launch_segments(segs, hp, s))) return st;
    }
    for (int i = 0; i < g->n_slots; ++i) {
        jnx_head_opt& o = opt[g->h_slot_tenant[i]];
        ++o.step;
        ++o.version;
    }
    return JNX_OK;
}
