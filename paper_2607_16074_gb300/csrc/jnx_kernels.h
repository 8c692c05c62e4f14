// Internal kernel launchers shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <vector>

#include "jnx_host.h"

namespace jnx {

enum { EPI_BF16 = 0, EPI_F32 = 1, EPI_RESID = 2, EPI_GLU = 3, EPI_ROPE = 4, EPI_GLU_BWD = 5,
       EPI_GLU_SAVE = 6, EPI_GLU_DM = 7 };

struct GemmParams {
    int M, N, K;
    int epi;
    void* out;            // EPI_BF16 / EPI_F32 / EPI_GLU / EPI_ROPE output
    int ldo;              // its row stride in elements
    float* resid;         // EPI_RESID: fp32 [M, ldr], updated in place
    int ldr;
    const int* pos;       // EPI_ROPE: position of each row
    const float2* rope;   // EPI_ROPE: (cos, sin) table [hd/2][rope_ld], frequency-major
    int rope_ld;          // EPI_ROPE: positions per frequency row of the table (max_pos)
    int rope_cols;        // EPI_ROPE: columns [0, rope_cols) get RoPE
    int hd;               // EPI_ROPE: head dim (64, 128 or 256)
    int act;              // EPI_GLU: JNX_GLU_*
    int group_m;          // tile-order group size (row blocks)
    int* status;          // device status word
    // RMSNorm folded across two GEMMs.  EPI_RESID with norm_gamma set also
    // writes y = bf16(x_new * gamma[col]) to norm_out [M, N] and, per row and
    // 128-column block, the partial sum of x_new^2 to ss_out [M, N / 128].
    const uint16_t* norm_gamma;
    uint16_t* norm_out;
    float* ss_out;
    // EPI_ROPE / EPI_GLU with ss_in set: the A rows are such y, and each
    // output row is first scaled by rsqrt(sum of ss_in[row][0, ss_parts) /
    // ss_cols + ss_eps), the RMSNorm factor of the row (a per-row scale
    // commutes with the product).
    const float* ss_in;
    int ss_parts, ss_cols;
    float ss_eps;
    // EPI_GLU_SAVE: over the gate/up weights (as EPI_GLU), writes bf16
    // u act'(g) in the gate columns and act(g) in the up columns of out
    // [M, N] (EPI_GLU's packed order: 128-column blocks alternating gate and
    // up): what the GLU backward multiplies the incoming gradient by.
    // EPI_GLU_BWD: the GEMM computes dm = dloss/d(act(g) * u) for F columns;
    // aux [M, ldaux] holds what EPI_GLU_SAVE wrote, and out (same layout; it
    // may be aux itself) receives dg = dm u act'(g) in the gate columns and
    // du = dm act(g) in the up columns, bf16.
    const uint16_t* aux;
    int ldaux;
    // EPI_GLU_DM: over the gate/up weights (as EPI_GLU); aux [M, ldaux]
    // holds dm = dloss/d(act(g) * u) in the up columns of the packed order
    // (F column f at packed column 256 (f / 128) + 128 + f % 128), and out
    // (same layout; it may be aux itself) receives dg = dm u act'(g) in the
    // gate columns and du = dm act(g) in the up columns, bf16.
    // EPI_BF16 with pack_up set writes output column n to packed column
    // 256 (n / 128) + 128 + n % 128 (dm into the up columns for EPI_GLU_DM).
    int pack_up;
};

constexpr int kMaxRopePos = 1 << 16;  // longest sample a workspace reserves RoPE rows for

// Argument checks shared by the backbone's entry points.
jnx_status check_backbone(const jnx_backbone* bb);
jnx_status check_group(const jnx_group* g);

// LoRA: rank and the number of tenant segments one launch describes.
constexpr int kLoraRank = 16;
constexpr int kLoraMaxSlots = 256;

// Per-tenant LoRA up-projection done on the tensor core inside a projection
// GEMM (EPI_ROPE or EPI_RESID): the GEMM's 128-row tiles are laid out per
// tenant segment (a tile never holds two tenants), and after the K loop of a
// tile one more K = 16 MMA adds t[rows, part] . B_part[tenant][cols]^T, where
// the tile's 256 output columns lie in one part (Q, K or V for the fused
// projection, the single part for O).
struct LoraGemm {
    CUtensorMap tt;          // t [M, ldt] bf16, box 16 x 128, 32-byte swizzle
    CUtensorMap tb[3];       // B_p viewed as [n_tenants * cols_p, 16], box 16 x 256
    int part_cols[3];        // output columns of each part (multiples of 256)
    int n_parts, n_seg;      // n_parts = 0: no up-projection (gemm_launch_seg)
    int seg_b;               // B holds every tenant's [N, K] weights stacked: a
                             // segment's tiles read rows seg_tenant * N + ...
    int seg_r0[kLoraMaxSlots], seg_r1[kLoraMaxSlots], seg_tenant[kLoraMaxSlots];
    int seg_tile0[kLoraMaxSlots + 1];  // first 128-row tile of each segment
};

// Host description of a LoRA up-projection for gemm_launch_lora.
struct LoraSpec {
    const uint16_t* t;       // [M, ldt] bf16 down-projected rows
    int ldt;
    const uint16_t* b[3];    // per part: [n_tenants, cols_p, r] bf16
    int cols[3];
    int n_parts, n_tenants;
    int n_seg;
    const int* seg_r0;       // host arrays [n_seg]: token rows of each tenant segment
    const int* seg_r1;
    const int* seg_tenant;
};

jnx_status gemm_launch_lora(const uint16_t* A, int lda, const uint16_t* B, int ldb, GemmParams p,
                            const LoraSpec& ls, cudaStream_t s);

// Segmented GEMM with per-tenant weights: for every segment i (rows
// [seg_r0[i], seg_r1[i]) of A and C, host arrays), C = A . B_t^T with B_t the
// [N, K] slice of tenant seg_tenant[i] in B = [n_tenants * N, K] (row stride
// ldb).  Output tiles never straddle two segments.  Any epilogue.
jnx_status gemm_launch_seg(const uint16_t* A, int lda, const uint16_t* B, int ldb, int n_tenants,
                           GemmParams p, int n_seg, const int* seg_r0, const int* seg_r1,
                           const int* seg_tenant, cudaStream_t s);
struct LoraSlots {
    int g0, n, sample0, pad_;
    int tenant[kLoraMaxSlots];
    int r0[kLoraMaxSlots], r1[kLoraMaxSlots], tile_start[kLoraMaxSlots];
};
struct LoraDown {
    const uint16_t* a[3];  // per part: [n_tenants, r, K]
};
// t[row, :] = bf16(x[row, :] . [A_0 | .. | A_{n_parts-1}][tenant(row)]^T).
jnx_status lora_down_launch(const jnx_group* g, const uint16_t* x, int ldx, int K, int n_parts,
                            const uint16_t* const* a, uint16_t* t, int ldt, cudaStream_t s);

// GEMM C = A . B^T with A [M, K] (row stride lda), B [N, K] (row stride ldb).
jnx_status gemm_check(int M, int N, int K);
jnx_status gemm_launch(const uint16_t* A, int lda, const uint16_t* B, int ldb, GemmParams p,
                       cudaStream_t s, int max_ctas = 0);
bool make_tmap_bf16(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols,
                    uint64_t row_stride_elems, uint32_t box_rows, uint32_t box_cols,
                    int swizzle_bytes = 128);
int num_sms();

// Raise fn's dynamic shared-memory limit to `bytes` on the current device,
// once per device (the attribute is per device; `done` holds one bit per
// device ordinal < 64, and callers that race both set it, which is harmless).
cudaError_t set_smem_limit(const void* fn, int bytes, std::atomic<uint64_t>& done);

// Packer: x[N, d] fp32 = widened gather of vision rows / text-embedding rows.
jnx_status pack_launch(const jnx_group* g, const uint16_t* vision, int64_t n_vision,
                       const int32_t* text_ids, int64_t n_text, const uint16_t* table, int vocab,
                       int d, float* x, int* status, cudaStream_t s);

// RMSNorm: out[M, d] bf16 = x / sqrt(mean(x^2) + eps) * gamma.
jnx_status rmsnorm_launch(const float* x, const uint16_t* gamma, float eps, int M, int d,
                          uint16_t* out, cudaStream_t s);

// Final RMSNorm fused with the per-sample mean pool.
jnx_status final_pool_launch(const float* x, const uint16_t* gamma, float eps, const int* cu,
                             int S, int d, float* pooled, uint16_t* hidden, cudaStream_t s);

// Folded RMSNorm, first half: y = bf16(x * gamma) [M, d] and per row and
// 128-column block the sum of x^2 (ss [M, d / 128]).
jnx_status rms_prep_launch(const float* x, const uint16_t* gamma, int M, int d, uint16_t* y,
                           float* ss, cudaStream_t s);

// (cos, sin) table for positions [0, max_pos) of head dim hd.
jnx_status rope_table_launch(float2* tab, int max_pos, int hd, float theta, cudaStream_t s);

// Varlen attention confined to each sample, bidirectional.  `items`
// (device, optional) lists the (sample, 128-query tile) work items in the
// order the persistent kernel should take them; null enumerates them.
// With lse set, also writes each query row's log2-sum-exp of its scaled
// scores, lse[row * H + h] = log2(sum_j 2^(s_j log2(e) / sqrt(hd))), which
// the backward uses to recompute the probabilities.
// Attention work items (sample, 128-row tile) of a group, most expensive first.
jnx_status build_attn_items(const jnx_group* g, std::vector<int2>& sorted);
// JNX_ERR_UNSUPPORTED when s is capturing into a CUDA graph (for the calls
// that upload a work list from host memory).
jnx_status refuse_capture(cudaStream_t s, const char* what);
// The attention work list for g: its own device copy if it has one, else
// uploaded into `upload` (refused on a capturing stream).
jnx_status attn_items_for(const jnx_group* g, int2* upload, cudaStream_t s, const char* what,
                          const int2*& items, int& n_items);

jnx_status attention_launch(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv, int hd,
                            const int* cu, int S, int max_seqlen, const int2* items, int n_items,
                            uint16_t* out, int ldo, float* lse, int* status, cudaStream_t s);

}  // namespace jnx
