// Internal descriptors for the tenant-head kernels.
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "jnx_host.h"

namespace jnx {

// One group slot: the tenant's head parameters and gradient buffers, and the
// packed-sample range [s0, s1) of that tenant.
struct HeadSlot {
    const uint16_t *w1, *b1, *w2, *b2;
    float *g_w1, *g_b1, *g_w2, *g_b2;
    int s0, s1;
    int d_in, d_hidden, width, tenant;
};

// Slots passed by value in kernel parameter space (up to kMaxSlots at once).
constexpr int kMaxSlots = 64;
struct HeadTable {
    HeadSlot slot[kMaxSlots];
};

// Head activations kept in the workspace between forward and backward;
// every array is [n_samples, ld] fp32 with ld >= max(d_hidden, width).
struct HeadScratch {
    float *z, *a, *y, *dy, *dz;
    int ld;
};

jnx_status mlp_heads_forward(const HeadTable& tab, int n, int max_hidden, int max_width,
                             const float* pooled, int d, const int* sample_target,
                             const float* targets, float* preds, float* loss, HeadScratch ws,
                             cudaStream_t s);
jnx_status mlp_heads_backward(const HeadTable& tab, int n, int max_hidden, int max_width,
                              int max_din, const float* pooled, int d, HeadScratch ws,
                              cudaStream_t s);

}  // namespace jnx
