// Internal kernel launchers shared by the library's translation units.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "jnx_host.h"

namespace jnx {

enum { EPI_BF16 = 0, EPI_F32 = 1, EPI_RESID = 2, EPI_GLU = 3, EPI_ROPE = 4 };

struct GemmParams {
    int M, N, K;
    int epi;
    void* out;            // EPI_BF16 / EPI_F32 / EPI_GLU / EPI_ROPE output
    int ldo;              // its row stride in elements
    float* resid;         // EPI_RESID: fp32 [M, ldr], updated in place
    int ldr;
    const int* pos;       // EPI_ROPE: position of each row
    const float2* rope;   // EPI_ROPE: (cos, sin) table [max_pos, hd/2]
    int rope_cols;        // EPI_ROPE: columns [0, rope_cols) get RoPE
    int hd;               // EPI_ROPE: head dim (64, 128 or 256)
    int act;              // EPI_GLU: JNX_GLU_*
    int group_m;          // tile-order group size (row blocks)
    int* status;          // device status word
    // LoRA up-projection (EPI_ROPE / EPI_RESID): when lora_t is set, the
    // epilogue adds t[row, p*r .. p*r+r) . B_p[tenant(row)][col', :] to each
    // column of part p before its own op.  Parts are consecutive column
    // ranges of lora_cols[p] columns; B_p is [n_tenants, lora_cols[p], r].
    const float* lora_t;  // [M, ldt] fp32
    int ldt;
    const int* row_tenant;
    const uint16_t* lora_b[3];
    int lora_cols[3];
};

// LoRA: rank and the number of tenant segments one launch describes.
constexpr int kLoraRank = 16;
constexpr int kLoraMaxSlots = 256;
struct LoraSlots {
    int g0, n, sample0, pad_;
    int tenant[kLoraMaxSlots];
    int r0[kLoraMaxSlots], r1[kLoraMaxSlots], tile_start[kLoraMaxSlots];
};
struct LoraDown {
    const uint16_t* a[3];  // per part: [n_tenants, r, K]
};
// row_tenant[r] for every packed row.
jnx_status lora_row_tenant_launch(const jnx_group* g, int* row_tenant, cudaStream_t s);
// t[row, :] = x[row, :] . [A_0 | .. | A_{n_parts-1}][tenant(row)]^T, fp32.
jnx_status lora_down_launch(const jnx_group* g, const uint16_t* x, int ldx, int K, int n_parts,
                            const uint16_t* const* a, float* t, int ldt, cudaStream_t s);

// GEMM C = A . B^T with A [M, K] (row stride lda), B [N, K] (row stride ldb).
jnx_status gemm_check(int M, int N, int K);
jnx_status gemm_launch(const uint16_t* A, int lda, const uint16_t* B, int ldb, GemmParams p,
                       cudaStream_t s, int max_ctas = 0);
bool make_tmap_bf16(CUtensorMap* m, const void* ptr, uint64_t rows, uint64_t cols,
                    uint64_t row_stride_elems, uint32_t box_rows, uint32_t box_cols);
int num_sms();

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

// (cos, sin) table for positions [0, max_pos) of head dim hd.
jnx_status rope_table_launch(float2* tab, int max_pos, int hd, float theta, cudaStream_t s);

// Varlen attention confined to each sample, bidirectional.
jnx_status attention_launch(const uint16_t* qkv, int ldq, int n_tokens, int H, int Hkv, int hd,
                            const int* cu, int S, int max_seqlen, uint16_t* out, int ldo,
                            int* status, cudaStream_t s);

}  // namespace jnx
