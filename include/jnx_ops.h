/*
 * Stage-level entry points of libjnx.so: each step of jnx_backbone_forward
 * on its own, for stage-wise parity tests and per-kernel measurement.  The
 * conventions of jnx.h apply (borrowed pointers, asynchronous on `stream`,
 * host-checked arguments, bf16 as uint16_t bit patterns, row-major).
 */
#ifndef JNX_OPS_H
#define JNX_OPS_H

#include "jnx.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Epilogues of jnx_op_gemm. */
#define JNX_EPI_BF16 0  /* out bf16 [M, ldo] = C */
#define JNX_EPI_F32 1   /* out fp32 [M, ldo] = C */
#define JNX_EPI_RESID 2 /* out fp32 [M, ldo] += C (residual stream update) */
#define JNX_EPI_GLU 3   /* W holds 128-row blocks alternating gate / up rows;
                           out bf16 [M, ldo] columns j < N/2 = act(C_gate) * C_up */
#define JNX_EPI_ROPE 4  /* out bf16 [M, ldo] = C with rotate-half RoPE at
                           position pos[row] on columns < rope_cols */
#define JNX_EPI_GLU_SAVE 6 /* W as for JNX_EPI_GLU; out bf16 [M, ldo], N columns in W's
                              packed order: u act'(g) in each gate column, act(g) in each
                              up column (the GLU backward's multipliers) */

/* The canonical packing step (§4.3: the VLAFeature is where the tenants'
 * samples are concatenated): x[t, :] = fp32 of vision[gather_src[t]] or of
 * text_table[text_ids[-gather_src[t] - 1]].  x is [n_tokens, d] fp32.  A
 * source index outside its buffer or a text id outside [0, vocab) writes a
 * zero row and JNX_ERR_DEVICE_BOUNDS to *status (device int, may be NULL). */
jnx_status jnx_op_pack(const jnx_group* g, const uint16_t* vision, int64_t n_vision_rows,
                       const int32_t* text_ids, int64_t n_text, const uint16_t* text_table,
                       int32_t vocab, int32_t d, float* x, int32_t* status, void* stream);

/* out[M, d] bf16 = x / sqrt(mean(x^2) + eps) * gamma, fp32 statistics;
 * d in {256, 512, 1024, 2048, 4096}. */
jnx_status jnx_op_rmsnorm(const float* x, const uint16_t* gamma, float eps, int32_t M, int32_t d,
                          uint16_t* out, void* stream);

/* Workspace bytes of jnx_op_gemm with JNX_EPI_ROPE for positions < max_pos. */
size_t jnx_op_gemm_workspace_bytes(int32_t max_pos, int32_t head_dim);

/* C[M, N] = A[M, K] W[N, K]^T on the tcgen05 tensor cores, fp32 accumulate,
 * then the epilogue.  N % 256 == 0, K % 64 == 0, A/W rows 16-byte aligned.
 * out has rows of ldo elements (bf16, or fp32 for JNX_EPI_F32 / RESID),
 * ldo >= the output width (N, or N / 2 for JNX_EPI_GLU), 16-byte aligned
 * rows and base, else JNX_ERR_INVALID_ARG.
 * pos/max_pos/rope_cols/head_dim/rope_theta are read for JNX_EPI_ROPE only
 * (workspace then holds the status word and the RoPE table; rope_cols a
 * multiple of head_dim within [0, N]; a position outside [0, max_pos) leaves
 * its row unrotated and records JNX_ERR_DEVICE_BOUNDS in the status word,
 * read by jnx_check_status(workspace)); act
 * (JNX_GLU_*) for JNX_EPI_GLU only.  workspace may be NULL otherwise. */
jnx_status jnx_op_gemm(const uint16_t* A, const uint16_t* W, int32_t M, int32_t N, int32_t K,
                       int32_t epilogue, void* out, int32_t ldo, const int32_t* pos,
                       int32_t max_pos, int32_t rope_cols, int32_t head_dim, float rope_theta,
                       int32_t act, void* workspace, size_t ws_bytes, void* stream);

/* Attention confined to each sample: for every sample s, head h,
 * out[t] = softmax(q_t K_s^T / sqrt(hd)) V_s over the sample's own tokens.
 * qkv [n_tokens, (H + 2 Hkv) hd] bf16 (q heads, then k heads, then v heads),
 * out [n_tokens, H hd] bf16; head_dim in {64, 128, 256}.  A wait that ran
 * out of time writes JNX_ERR_TIMEOUT to *status (device int, may be NULL). */
jnx_status jnx_op_attention(const uint16_t* qkv, int32_t n_tokens, int32_t n_heads,
                            int32_t n_kv_heads, int32_t head_dim, const int32_t* cu_seqlens,
                            int32_t n_samples, int32_t max_seqlen, uint16_t* out,
                            int32_t* status, void* stream);

/* Final RMSNorm and per-sample mean: pooled[s] = gamma * mean over the
 * sample's rows of x_t / sqrt(mean(x_t^2) + eps) (fp32), hidden[t] = bf16
 * of the normed row.  Either output may be NULL. */
jnx_status jnx_op_final_pool(const float* x, const uint16_t* gamma, float eps,
                             const int32_t* cu_seqlens, int32_t n_samples, int32_t d,
                             float* pooled, uint16_t* hidden, void* stream);

/* ---- stages of the adapter backward (jnx_backbone_backward_lora) ---- */

/* jnx_op_attention that also writes lse [n_tokens, H] fp32: each query
 * row's log2-sum-exp of its scaled scores, log2(sum_j 2^(s_j log2(e) /
 * sqrt(hd))), from which the backward recomputes the probabilities. */
jnx_status jnx_op_attention_lse(const uint16_t* qkv, int32_t n_tokens, int32_t n_heads,
                                int32_t n_kv_heads, int32_t head_dim, const int32_t* cu_seqlens,
                                int32_t n_samples, int32_t max_seqlen, uint16_t* out, float* lse,
                                int32_t* status, void* stream);

/* The attention backward's prologue: dO [n_tokens, H hd] bf16 = bf16(datt)
 * (fp32) and D [n_tokens, H] = per head, the sum over its hd columns of
 * dO * att (att = the forward's output, bf16). */
jnx_status jnx_op_attention_backward_prep(const float* datt, const uint16_t* att, int32_t n_tokens,
                                          int32_t n_heads, int32_t head_dim, uint16_t* dO,
                                          float* D, void* stream);

/* Workspace bytes of jnx_op_attention_backward. */
size_t jnx_op_attention_backward_workspace_bytes(int32_t n_tokens, int32_t max_seqlen,
                                                 int32_t head_dim);

/* Gradients of jnx_op_attention with respect to its input qkv, given dO,
 * the forward's lse and D (jnx_op_attention_backward_prep): for query head
 * h on K/V head g, P = softmax(q k^T / sqrt(hd)) inside each sample,
 * dv_g += P^T dO_h, dS = P * (dO_h v_g^T - D), dq_h = dS k_g / sqrt(hd),
 * dk_g += dS^T q_h / sqrt(hd).  qkv holds q and k after RoPE; dqkv
 * [n_tokens, (H + 2 Hkv) hd] bf16 receives the gradients of the pre-RoPE
 * projections (dq, dk rotated back by the rotate-half RoPE of theta at
 * pos[t]; dv as is).  h_cu_seqlens is the host copy of cu_seqlens (the work
 * list is built from it).  A wait that ran out of time writes
 * JNX_ERR_TIMEOUT to *status. */
jnx_status jnx_op_attention_backward(const uint16_t* qkv, const uint16_t* dO, const float* lse,
                                     const float* D, int32_t n_tokens, int32_t n_heads,
                                     int32_t n_kv_heads, int32_t head_dim,
                                     const int32_t* cu_seqlens, const int32_t* h_cu_seqlens,
                                     int32_t n_samples, int32_t max_seqlen, const int32_t* pos,
                                     float rope_theta, uint16_t* dqkv, void* workspace,
                                     size_t ws_bytes, int32_t* status, void* stream);

/* RMSNorm backward: with s = rsqrt(mean(x^2) + eps) per row,
 * dx = dres + s gamma dn - x s^3 mean(gamma dn x) (fp32; dres may be NULL
 * or dx itself) and dx_bf = bf16(dx) when not NULL.  d % 128 == 0. */
jnx_status jnx_op_rms_backward(const float* x, const uint16_t* gamma, float eps, const float* dn,
                               const float* dres, int32_t M, int32_t d, float* dx,
                               uint16_t* dx_bf, void* stream);

/* The feed-forward backward's first GEMM with the GLU backward fused:
 * dm[M, F] = A[M, K] W[F, K]^T is the gradient at act(g) * u; gu [M, 2F]
 * bf16 holds on entry what JNX_EPI_GLU_SAVE wrote (u act'(g) in the gate
 * columns, act(g) in the up columns of the packed order, 128-column blocks
 * alternating gate and up) and on return dg = dm u act'(g) in the gate
 * columns, du = dm act(g) in the up columns.  F % 256 == 0, K % 64 == 0.
 * act is not read (the multipliers already hold the activation). */
jnx_status jnx_op_gemm_glu_backward(const uint16_t* A, const uint16_t* W, int32_t M, int32_t F,
                                    int32_t K, uint16_t* gu, int32_t act, void* stream);

/* The feed-forward backward's GLU step with the gate/up GEMM recomputed
 * (what jnx_backbone_backward_lora runs per block): dm[M, F] = dy[M, d]
 * w_down_t[F, d]^T is the gradient at act(g) * u; it is stored bf16 in the
 * up columns of gu [M, 2F] (packed order: 128-column blocks alternating
 * gate and up), then the gate/up GEMM g|u = n2[M, d] w_gu[2F, d]^T (w_gu in
 * the packed order of jnx_pack_gate_up) leaves dg = dm u act'(g) in the gate
 * columns and du = dm act(g) in the up columns, bf16.  gu needs no content
 * on entry.  F % 256 == 0 (the GEMM's 256-column tiles), d % 64 == 0, gu
 * 16-byte aligned, act a JNX_GLU_* value (JNX_ERR_INVALID_ARG otherwise). */
jnx_status jnx_op_ffn_glu_backward(const uint16_t* dy, const uint16_t* w_down_t,
                                   const uint16_t* n2, const uint16_t* w_gu, int32_t M, int32_t F,
                                   int32_t d, int32_t act, uint16_t* gu, void* stream);

/* The fused QKV projection + RoPE of jnx_op_gemm (JNX_EPI_ROPE) for callers
 * that cannot allocate device memory — e.g. a plugin in a serving process
 * whose pool owns every device allocation, or a batching worker that must
 * not call cudaMalloc between requests because it can stall the device.
 * The paper has no counterpart: this is a deployment variant of the library.
 * The caller passes inputs and outputs only; the status word and the RoPE
 * table live in a fixed file-scope device array inside the library (every
 * GPU that loads the library holds it until exit; nothing is allocated).
 * Limits: max_pos * head_dim / 2 <= JNX_NOALLOC_MAX_ROPE_ENTRIES, otherwise
 * JNX_ERR_UNSUPPORTED before any launch.  Host-detected errors (null
 * pointers, head_dim not 64/128/256, rope_cols not a multiple of head_dim
 * within [0, N], ldo < N, out or its rows not 16-byte aligned) return
 * JNX_ERR_INVALID_ARG before any launch with nothing written.  A position
 * outside [0, max_pos) is a device-detected error: its row is written
 * unrotated and JNX_ERR_DEVICE_BOUNDS is recorded in the array's status
 * word (read it with jnx_op_gemm_rope_noalloc_status).
 * The first call on a device looks up the array's address (make it before
 * any stream capture).  All calls on a device share the array: each clears
 * the status word and rewrites the table it reads, and calls that overlap on
 * the GPU race.  Arguments and results otherwise as jnx_op_gemm. */
#define JNX_NOALLOC_MAX_ROPE_ENTRIES (1 << 19)
jnx_status jnx_op_gemm_rope_noalloc(const uint16_t* A, const uint16_t* W, int32_t M, int32_t N,
                                    int32_t K, uint16_t* out, int32_t ldo, const int32_t* pos,
                                    int32_t max_pos, int32_t rope_cols, int32_t head_dim,
                                    float rope_theta, void* stream);

/* Reads and clears the status word of jnx_op_gemm_rope_noalloc's fixed
 * array on the current device, after the work queued on `stream` (it
 * synchronises the stream; allocates nothing).  Returns JNX_OK, or the
 * first error a kernel recorded since the last read or call (a call clears
 * it on entry): JNX_ERR_DEVICE_BOUNDS, JNX_ERR_TIMEOUT. */
jnx_status jnx_op_gemm_rope_noalloc_status(void* stream);

/* Diagnostics: two device routines of the hot path run on their own, so
 * tests can pin them.  Neither is part of the grouped path.
 *
 * y[i] = 2^x[i] by the polynomial exponential that the varlen attention's
 * softmax evaluates for one key pair in four (range reduction j = rint(x),
 * f = x - j, 2^f by the degree-3 minimax polynomial on [-0.5, 0.5], x
 * clamped at -126).  x, y: n device floats.  It stands for the softmax
 * probabilities 2^(s - m) of §5.2's shared backbone attention. */
jnx_status jnx_diag_ex2_poly(const float* x, float* y, int32_t n, void* stream);

/* One thread waits, through the library's bounded mbarrier wait, on a
 * barrier that completes (arrive != 0) or that nothing ever arrives on
 * (arrive == 0), giving up after limit_cycles SM clocks (0 < limit <= 2^31,
 * else JNX_ERR_INVALID_ARG before the launch).  A wait that gave up writes
 * JNX_ERR_TIMEOUT to *status (a device int) and the kernel returns; every
 * spin in the library's kernels behaves this way.  The paper has no
 * counterpart (failure detection of the kernels themselves). */
jnx_status jnx_diag_bounded_wait(int64_t limit_cycles, int32_t arrive, int32_t* status,
                                 void* stream);

#ifdef __cplusplus
}
#endif

#endif /* JNX_OPS_H */
