// Internal launchers of the per-tenant LoRA backward (bwd.cu, attn_bwd.cu).
#pragma once
#include <cuda_runtime.h>
#include <stdint.h>

#include "jnx_host.h"

namespace jnx {

constexpr int kSegMaxSlots = 256;    // tenant segments one launch describes
constexpr int kSegMaxChunks = 1024;  // row chunks of an adapter-gradient launch
constexpr int kSegChunkRows = 1024;  // shortest row chunk

// Token rows of each group tenant (its contiguous packed segment), cut into
// tiles of `bm` rows that never straddle two tenants.
struct SegRows {
    int n;
    int tenant[kSegMaxSlots];
    int r0[kSegMaxSlots], r1[kSegMaxSlots], tile_start[kSegMaxSlots];
};

// Up to four summed parts of a segmented up-projection: T_p [rows, k_p]
// (row stride ldt_p, bf16) times the group slot's W_p, row-major
// [k_p, ncols] bf16.  A slot whose W_0 is null is skipped (its rows are not
// written).
struct SegUpParts {
    const uint16_t* t[4];
    int ldt[4];
    int k[4];
    int n_parts;
    const uint16_t* w[4][kSegMaxSlots];
};

// W_p of every group slot = base_p + tenant * stride_p (an adapter array
// [n_tenants, k_p, ncols]).
void seg_up_weights(const jnx_group* g, SegUpParts& sp, int part, const uint16_t* base,
                    long long stride);

// Row chunks of the group's tenant segments for the adapter gradients.
struct SegChunks {
    int n_slots;
    int slot_tenant[kSegMaxSlots];
    int slot_chunk0[kSegMaxSlots + 1];
    int r0[kSegMaxChunks], r1[kSegMaxChunks];
};

// MLP first-layer weights per group slot (null for a query-head slot).
struct MlpFeatTable {
    const uint16_t* w1[kSegMaxSlots];
    int hid[kSegMaxSlots];
};

jnx_status transpose_launch(const uint16_t* src, int batch, int rows, int cols, uint16_t* dst,
                            cudaStream_t s);
jnx_status rms_bwd_launch(const float* x, const uint16_t* gamma, float eps, const float* dn,
                          const float* dres, int M, int d, float* dx, uint16_t* dx_bf,
                          cudaStream_t s);
jnx_status attn_bwd_prep_launch(const float* datt, const uint16_t* att, int M, int H, int hd,
                                uint16_t* dO, float* D, cudaStream_t s);
jnx_status seg_rows_build(const jnx_group* g, int bm, SegRows& sr, int& tiles);
// out[rows of tenant t, :ncols] (+)= sum_p T_p W_p[t]
jnx_status seg_up_launch(const jnx_group* g, const SegUpParts& sp, int ncols, float* out, int ldo,
                         bool add, cudaStream_t s);
// Floats of the partial-sum buffer seg_tn_launch needs.
size_t seg_tn_part_floats(int n_tokens, int n_slots, int n);
// For every group tenant t: G = U_t^T V_t over its rows (U [rows, 16],
// V [rows, n]) written or added to grad + t * gstride as [16, n] or, with
// trans, [n, 16].
jnx_status seg_tn_launch(const jnx_group* g, const uint16_t* U, int ldu, const uint16_t* V,
                         int ldv, int n, float* part, size_t part_floats, float* grad,
                         long long gstride, bool trans, bool add, cudaStream_t s);
// For every segment i of sr (rows [r0, r1), tenant): G[tenant][m, n] = (or
// +=) sum over the rows of U[row, m] V[row, n]; m % 64 == 0, n % 128 == 0.
// dst [cols][kpad] bf16: segment i's rows of src [*, ld_src] transposed to
// columns sr.tile_start[i] .. (64-aligned, ascending), zero elsewhere.
jnx_status transpose_seg_launch(const uint16_t* src, int ld_src, int cols, const SegRows& sr,
                                int kpad, uint16_t* dst, cudaStream_t s);
jnx_status seg_wgrad_launch(const SegRows& sr, const uint16_t* U, int ldu, const uint16_t* V,
                            int ldv, int m, int n, float* grad, long long gstride, bool add,
                            cudaStream_t s);
jnx_status mlp_dfeat_launch(const float* dz, int ldz, const int* cu, const int* sample_slot,
                            int n_samples, const MlpFeatTable& tab, int d, float* dh,
                            cudaStream_t s);
jnx_status to_bf16_launch(const float* src, int lds, int rows, int cols, uint16_t* dst, int ldd,
                          cudaStream_t s);

// Attention backward over the packed samples (bidirectional inside each
// sample), from q, k, v (after RoPE, [N, (H + 2 Hkv) hd]), the saved
// log2-sum-exp lse [N, H] of the forward, dO [N, H hd] bf16 and
// D = rowsum(dO * O) [N, H].  Writes dq, dk, dv with the inverse RoPE
// applied to dq and dk (the gradients of the pre-RoPE projections) into
// dqkv [N, (H + 2 Hkv) hd] bf16.
jnx_status attention_bwd_launch(const uint16_t* qkv, int ldq, const uint16_t* dO, const float* lse,
                                const float* D, int n_tokens, int H, int Hkv, int hd,
                                const int* cu, const int* pos, const float2* rope, int rope_ld,
                                const int2* items, int n_items, uint16_t* dqkv, int* status,
                                cudaStream_t s);

}  // namespace jnx
