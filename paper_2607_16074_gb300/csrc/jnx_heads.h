// Internal descriptors for the tenant-head kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "jnx_host.h"

namespace jnx {

// One group slot: the tenant's head parameters and gradient buffers, its
// packed samples [s0, s1) and token rows [r0, r1).
struct HeadSlot {
    int kind;        // JNX_HEAD_MLP or JNX_HEAD_XATTN
    int tenant;
    int s0, s1;
    int r0, r1;
    int d_in;        // backbone width
    int hid;         // input width of the output layer: MLP d_hidden, query head nq * dq
    int width;       // outputs per sample
    int nq, dq;      // query head
    int accum;       // add into the gradient buffers instead of overwriting them
    const uint16_t *w1, *b1;   // MLP first layer
    const uint16_t *w2, *b2;   // output layer: MLP W2/b2 or query-head Wout/bout
    const uint16_t *q, *wk, *wv;
    float *g_w1, *g_b1, *g_w2, *g_b2, *g_q, *g_wk, *g_wv;
};

// Slots passed by value in kernel parameter space (up to kMaxSlots at once).
constexpr int kMaxSlots = 64;
struct HeadTable {
    HeadSlot slot[kMaxSlots];
};

// The fused optimizer step of the heads backward: per slot, the AdamW state
// of its 9 possible parameter tensors (jnx_head_opt order: w1, b1, w2, b2,
// q, wk, wv, wout, bout; the output layer's are 2, 3 for an MLP head and
// 7, 8 for a query head), the bf16 parameters it rewrites and the bias
// corrections of this step.
struct HeadOpt {
    float* master[9];
    float* m[9];
    float* v[9];
    uint16_t* p[9];
    float c1, c2;
};
struct HeadOptTable {
    HeadOpt slot[kMaxSlots];
};
struct AdamHp {
    float lr, b1, b2, eps, wd;
};

// What one launch batch of slots holds.
struct HeadBatch {
    int g0, n;                 // group slots [g0, g0 + n)
    int sample0, sample1;      // their packed samples
    int max_hid, max_mlp_hid, max_width, max_nq, max_dq;
    int max_ns;                // most samples in one slot
    bool any_mlp, any_xattn;
};

// Head activations kept in the workspace between forward and backward.
struct HeadScratch {
    float *z, *h, *dh;   // [n_samples, ld_h]
    float *y, *dy;       // [n_samples, ld_y]
    int ld_h, ld_y;
    // query heads
    float *kbuf, *vbuf, *dk, *dv;  // [n_tokens, ldkv]
    int ldkv;
    float *P, *dS;                 // [nq * n_tokens], key-major per sample
    float* dQs;                    // [n_samples, ld_h]
    float *Gs, *Hs;                // [n_samples, 32, d]: dS_s^T X_s and P_s^T X_s (32 query rows)
    uint16_t* dkv_bf;              // feature gradient: bf16 [dk | dv] rows [n_tokens, 2 ldkv]
};

jnx_status heads_forward_launch(const HeadTable& tab, const HeadBatch& b, const HeadScratch& ws,
                                const float* pooled, int d, const int* cu, const int* sample_slot,
                                const int* sample_target, const float* targets, float* preds,
                                float* loss, cudaStream_t s);
// kv_grads: also write the query heads' per-row dk, dv (read by the feature
// gradient only).
jnx_status heads_backward_launch(const HeadTable& tab, const HeadBatch& b, const HeadScratch& ws,
                                 const float* pooled, int d, const uint16_t* hidden,
                                 const int* cu, const int* sample_slot, bool kv_grads,
                                 cudaStream_t s);
// The backward with the tenant-private AdamW step fused into it, in two
// launches so that nothing updates a parameter before every read of it:
// front: the output layer's input gradient (reads W2 / Wout) and the query
// heads' attention backward (reads the learned queries); the caller may
// then form the feature gradient (reads W1, Wk, Wv); step: every
// parameter's gradient element goes straight into its AdamW update (plus
// the accumulated gradient buffer when the slots accumulate) and is not
// stored; the query heads' Wk/Wv kernel (reads the queries) runs before
// the queries' own update.
jnx_status heads_backward_front_launch(const HeadTable& tab, const HeadBatch& b,
                                       const HeadScratch& ws, int d, const uint16_t* hidden,
                                       const int* cu, const int* sample_slot, bool kv_grads,
                                       cudaStream_t s);
jnx_status heads_backward_step_launch(const HeadTable& tab, const HeadOptTable& opt,
                                      const AdamHp& hp, const HeadBatch& b,
                                      const HeadScratch& ws, const float* pooled, int d,
                                      cudaStream_t s);
jnx_status heads_set_smem();

}  // namespace jnx
