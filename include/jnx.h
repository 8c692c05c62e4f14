/*
 * jnx — grouped multi-tenant backbone forward with tenant-private action heads.
 *
 * C ABI of the GB300 (sm_103a) library libjnx.so.  The calls follow the
 * paper's statement of group batching:
 *
 *   jnx_group_plan        collect the largest FIFO-compatible prefix of
 *                         requests and canonicalise it into one packed varlen
 *                         batch with its slices (App. A, "Inference Queue
 *                         Composition"; §4.3, "Multi-Tenant Group Batching").
 *   jnx_backbone_forward  one shared frozen backbone forward over the packed
 *                         batch (the `encode` of App. A; §5.2 group execution).
 *   jnx_heads_forward     split the features by the recorded slices and run
 *                         each tenant's own action head and L2 loss on that
 *                         tenant's samples only (App. A `split`/`decode`;
 *                         §5.2 tenant-private loss).
 *   jnx_heads_backward    gradients of each tenant's loss into that tenant's
 *                         slot only; nothing is summed across tenants
 *                         (App. A, "Actor Consumption and Version
 *                         Consistency"; §5.2 tenant-private backward).
 *
 * Conventions for every call:
 *   - All pointers are borrowed.  The library allocates no device memory and
 *     frees nothing; scratch space is the caller's `workspace`.
 *   - Device calls are asynchronous on `stream` (a cudaStream_t passed as
 *     void*; NULL = the legacy default stream).
 *   - Arguments the host can check are checked before any launch; on error
 *     nothing is written and a message is available from jnx_last_error().
 *   - Errors a kernel detects (an index outside its buffer) set a status word
 *     at the start of the workspace instead of faulting; the offending access
 *     is skipped.  jnx_check_status() reads and clears it.
 *   - bf16 arrays are passed as uint16_t bit patterns; all matrices are
 *     row-major, projections stored [out, in].
 */
#ifndef JNX_H
#define JNX_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int32_t jnx_status;

#define JNX_OK 0
#define JNX_ERR_INVALID_ARG (-1)
#define JNX_ERR_CAPACITY (-3)
#define JNX_ERR_OVERFLOW (-5)
#define JNX_ERR_CUDA (-6)
#define JNX_ERR_DEVICE_BOUNDS (-7)
#define JNX_ERR_TIMEOUT (-8)
#define JNX_ERR_UNSUPPORTED (-9)
#define JNX_ERR_WORKSPACE (-10)

/* Message describing the last error returned on this thread ("" if none). */
const char* jnx_last_error(void);

/* Library ABI version (increments on any struct or signature change). */
int32_t jnx_version(void);

/* ------------------------------------------------------------------------
 * Plan (host only; callable without a GPU)
 * ------------------------------------------------------------------------ */

/* A tenant schema.  The first six fields are the shared-prefix signature:
 * two requests are compatible iff these are equal ("compatibility is
 * determined at the shared frozen-prefix boundary rather than by tenant
 * identity", App. A).  max_images and action_width describe the tenant's
 * own input limit and output structure and do not affect compatibility. */
typedef struct {
    int32_t backbone_id;
    int32_t d_model;
    int32_t vision_tokens;  /* rows per image */
    int32_t embed_dtype;    /* 0 = bf16 */
    int32_t vocab_id;
    int32_t rope_id;
    int32_t max_images;     /* per sample */
    int32_t action_width;   /* C * D_t floats per sample (targets, predictions) */
} jnx_schema;

/* One sample (observation) of a request.  Its vision rows are
 * vision[vision_row .. vision_row + n_img*vision_tokens), its text ids
 * text_ids[text_pos .. text_pos + text_len), its targets / predictions
 * targets[target_off .. target_off + action_width). */
typedef struct {
    int32_t n_img;
    int32_t text_len;
    int64_t vision_row;
    int64_t text_pos;
    int64_t target_off;
} jnx_sample;

/* One inference request in arrival order (App. A `InferenceRequest`). */
typedef struct {
    int32_t tenant;      /* tenant slot, 0 <= tenant < n_tenants */
    int32_t schema;      /* index into the schema array */
    int32_t n_samples;   /* >= 1 */
    int32_t reserved;
    const jnx_sample* samples;  /* [n_samples] */
} jnx_request;

typedef struct {
    int32_t max_samples;  /* batch limit in samples */
    int32_t max_tokens;   /* batch limit in packed tokens */
} jnx_limits;

/* Plan output: caller-owned host arrays with their capacities.
 *   cu_seqlens[S+1]   token offset of each packed sample
 *   sample_slot[S]    group slot (0..n_slots-1) of each packed sample
 *   sample_req[S]     index of the accepted request it came from
 *   sample_target[S]  its target/prediction offset (from jnx_sample)
 *   sample_width[S]   its action width (from its schema)
 *   seg_offsets[G+1]  packed-sample offsets of each group slot
 *   slot_tenant[G]    tenant of each group slot
 *   gather_src[N]     per packed token: vision row (>= 0) or
 *                     -(text position + 1) (< 0)
 *   pos_ids[N]        per packed token: position inside its sample
 * Packed order: tenants by first appearance, their requests in arrival
 * order, each request's samples in order; in a sample the vision rows of
 * its images first, then its text tokens.  Positions restart at 0. */
typedef struct {
    int32_t cap_samples, cap_tokens, cap_slots;  /* in */
    int32_t n_requests;                          /* out: accepted prefix length */
    int32_t n_samples, n_tokens, n_slots, max_seqlen;  /* out */
    int32_t* cu_seqlens;
    int32_t* sample_slot;
    int32_t* sample_req;
    int32_t* sample_target;
    int32_t* sample_width;
    int32_t* seg_offsets;
    int32_t* slot_tenant;
    int32_t* gather_src;
    int32_t* pos_ids;
} jnx_plan;

/* Collect the largest FIFO-compatible prefix of `reqs` and canonicalise it.
 * Scanning stops at the first request whose prefix signature differs from
 * the first request's, or that would push the batch over `lim` (whole
 * requests; the first request is always accepted so the queue drains).
 * Errors: JNX_ERR_INVALID_ARG (bad tenant/schema index, n_samples < 1, a
 * sample with n_img outside [0, max_images], text_len < 0 or no token),
 * JNX_ERR_OVERFLOW (a row, position or offset outside int32),
 * JNX_ERR_CAPACITY (arrays too small: the required n_samples, n_tokens and
 * n_slots are written back, nothing else).  n_reqs == 0 gives an empty plan. */
jnx_status jnx_group_plan(const jnx_schema* schemas, int32_t n_schemas,
                          const jnx_request* reqs, int32_t n_reqs, int32_t n_tenants,
                          const jnx_limits* lim, jnx_plan* out);

/* ------------------------------------------------------------------------
 * Inference scheduler (host only; callable without a GPU)
 * ------------------------------------------------------------------------ */

/* §4.3: the inference service has a maximum waiting time T and a target
 * batch size B; it builds a batch from requests in FIFO order and starts it
 * when the waiting time reaches T or the batch size reaches B. */
typedef struct {
    double timeout;         /* T, seconds the oldest queued request may wait */
    int32_t batch_samples;  /* B, in samples: a batch this large starts at once;
                               also the batch's sample limit */
    int32_t max_tokens;     /* packed-token limit of one batch */
    int32_t skip_ahead;     /* 0: stop at the first request incompatible with the
                               oldest (App. A prefix); 1: pass over such requests,
                               which stay queued, and take later compatible ones */
    int32_t reserved;
} jnx_sched_policy;

/* The scheduler's decision at time `now` over a queue of n_reqs requests in
 * arrival order (arrival[i] in seconds, any common origin).  It collects a
 * batch as jnx_group_plan does (requests compatible with the oldest one,
 * whole requests within batch_samples and max_tokens, the oldest always
 * taken) and fires when the batch holds >= batch_samples samples, when it
 * cannot grow (the next compatible request does not fit), or when the
 * oldest request has waited >= timeout.  Firing: *n_take > 0 and take[0..
 * *n_take) are the ascending queue indices to run (the caller removes them
 * from its queue and plans them with jnx_group_plan, which accepts them
 * all); *wake = now.  Not firing: *n_take = 0 and *wake = arrival[0] +
 * timeout, the time to poll again (HUGE_VAL for an empty queue).  take[]
 * holds n_reqs entries (caller-owned).  Errors: JNX_ERR_INVALID_ARG (null
 * pointer, a policy with batch_samples < 1, max_tokens < 1, timeout < 0 or
 * skip_ahead not 0/1, or a malformed request as jnx_group_plan rejects it),
 * JNX_ERR_OVERFLOW as jnx_group_plan; nothing is written on error. */
jnx_status jnx_sched_poll(const jnx_schema* schemas, int32_t n_schemas,
                          const jnx_request* reqs, const double* arrival, int32_t n_reqs,
                          int32_t n_tenants, double now, const jnx_sched_policy* pol,
                          int32_t* take, int32_t* n_take, double* wake);

/* ------------------------------------------------------------------------
 * Device-side view of a plan
 * ------------------------------------------------------------------------ */

/* The plan arrays copied to the device (the caller copies them), plus the
 * host copies the launcher reads to shape its launches. */
typedef struct {
    int32_t n_samples, n_tokens, n_slots, max_seqlen;
    const int32_t* cu_seqlens;     /* device [n_samples + 1] */
    const int32_t* sample_slot;    /* device [n_samples] */
    const int32_t* sample_target;  /* device [n_samples] */
    const int32_t* seg_offsets;    /* device [n_slots + 1] */
    const int32_t* gather_src;     /* device [n_tokens] */
    const int32_t* pos_ids;        /* device [n_tokens] */
    const int32_t* h_cu_seqlens;   /* host   [n_samples + 1] */
    const int32_t* h_seg_offsets;  /* host   [n_slots + 1] */
    const int32_t* h_slot_tenant;  /* host   [n_slots] */
    /* Optional: the group's attention work list on the device, [n_attn_items]
     * (sample, 128-row tile) int32 pairs exactly as jnx_group_attn_items
     * writes them, 8-byte aligned.  When it is set, the backbone forward and
     * backward read it instead of uploading their own copy, which makes them
     * capturable into a CUDA graph; NULL (and 0) keeps the upload. */
    const int32_t* attn_items;
    int32_t n_attn_items;
} jnx_group;

/* The group's attention work list on the host: (sample, 128-row tile) pairs,
 * the most expensive first, into out[2 * cap].  Returns the number of pairs;
 * when out is NULL or cap is smaller, writes nothing and returns that number
 * (call again with room); < 0 on an invalid group.  Needs n_samples,
 * n_tokens and h_cu_seqlens only. */
int32_t jnx_group_attn_items(const jnx_group* g, int32_t* out, int32_t cap);

/* ------------------------------------------------------------------------
 * Shared frozen backbone
 * ------------------------------------------------------------------------ */

#define JNX_GLU_SWIGLU 0     /* act = SiLU */
#define JNX_GLU_GEGLU_TANH 1 /* act = tanh-approximated GELU */

/* One pre-norm decoder block (device pointers, bf16):
 *   n1 = RMSNorm(x) * attn_norm;  [q|k|v] = n1 W_qkv^T; RoPE on q, k;
 *   x += W_o Attn(q, k, v);  n2 = RMSNorm(x) * ffn_norm;
 *   x += W_down (act(n2 W_g^T) * (n2 W_u^T)).
 * w_qkv  [(H + 2 Hkv) hd, d]: rows of W_q, then W_k, then W_v.
 * w_gu   [2 F, d]: 128-row blocks alternating gate and up rows, i.e. block
 *        2j holds gate rows 128j..128j+127 and block 2j+1 the matching up
 *        rows (jnx_pack_gate_up builds it from W_g and W_u).
 * LoRA (lora_rank r > 0): for each of q, k, v, o, per-tenant adapters
 *   lora_a_* [n_tenants, r, in] and lora_b_* [n_tenants, out, r];
 *   y += (x A_t^T) B_t^T for the rows of tenant t.  NULL when r == 0. */
typedef struct {
    const uint16_t* attn_norm;  /* [d] */
    const uint16_t* w_qkv;
    const uint16_t* w_o;        /* [d, H hd] */
    const uint16_t* ffn_norm;   /* [d] */
    const uint16_t* w_gu;
    const uint16_t* w_down;     /* [d, F] */
    const uint16_t* lora_a_q; const uint16_t* lora_b_q;
    const uint16_t* lora_a_k; const uint16_t* lora_b_k;
    const uint16_t* lora_a_v; const uint16_t* lora_b_v;
    const uint16_t* lora_a_o; const uint16_t* lora_b_o;
} jnx_layer;

typedef struct {
    int32_t n_layers, d_model, n_heads, n_kv_heads, head_dim, d_ff;
    int32_t glu;           /* JNX_GLU_* */
    int32_t lora_rank;     /* 0 = no adapters */
    int32_t n_tenants;     /* rows of the LoRA adapter arrays */
    int32_t vocab;
    int32_t vision_tokens;
    float eps;             /* RMSNorm epsilon */
    float rope_theta;
    const uint16_t* text_table;  /* device [vocab, d] */
    const uint16_t* final_norm;  /* device [d] */
    const jnx_layer* layers;     /* HOST array [n_layers] of device pointers */
} jnx_backbone;

/* Workspace bytes jnx_backbone_forward needs for a batch of n_tokens. */
size_t jnx_backbone_workspace_bytes(const jnx_backbone* bb, int32_t n_tokens);

/* Pack the batch (vision rows / text-embedding rows by gather_src), run all
 * blocks over it with attention confined to each sample, apply the final
 * RMSNorm and write the features:
 *   pooled [n_samples, d] fp32: the mean of each sample's final normed rows
 *          (features for MLP heads), or NULL;
 *   hidden [n_tokens, d] bf16: the final normed rows (features for query
 *          heads), or NULL.
 * vision [n_vision_rows, d] bf16 and text_ids [n_text] int32 are the
 * caller's observation buffers that gather_src indexes.  A gather index
 * outside them, or a text id outside [0, vocab), sets
 * JNX_ERR_DEVICE_BOUNDS in the status word and the row is zero-filled.
 * Without the group's attn_items the call uploads the attention work list
 * from host memory, which a CUDA graph cannot replay: on a capturing stream
 * it then returns JNX_ERR_UNSUPPORTED before any launch (as do
 * jnx_backbone_forward_train and jnx_backbone_backward_lora, and
 * jnx_op_attention_backward always).  With attn_items set the forward and
 * the backward are capturable. */
jnx_status jnx_backbone_forward(const jnx_backbone* bb, const jnx_group* g,
                                const uint16_t* vision, int64_t n_vision_rows,
                                const int32_t* text_ids, int64_t n_text,
                                float* pooled, uint16_t* hidden,
                                void* workspace, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Tenant-private action heads (one slot per tenant)
 * ------------------------------------------------------------------------ */

#define JNX_HEAD_MLP 0    /* y = SiLU(p W1^T + b1) W2^T + b2 on the pooled feature p */
#define JNX_HEAD_XATTN 1  /* y = flatten(softmax(Q k^T/sqrt(dq)) v) Wout^T + bout,
                             k = X Wk^T, v = X Wv^T over the sample's hidden rows X */

typedef struct {
    int32_t kind;       /* JNX_HEAD_* */
    int32_t d_in;       /* backbone width d */
    int32_t d_hidden;   /* MLP hidden width */
    int32_t n_queries;  /* query head: learned queries */
    int32_t q_dim;      /* query head: attention width */
    int32_t width;      /* outputs per sample, C * D_t */
    /* MLP (device, bf16): w1 [d_hidden, d_in], b1 [d_hidden], w2 [width, d_hidden], b2 [width] */
    const uint16_t *w1, *b1, *w2, *b2;
    /* query head (device, bf16): q [n_queries, q_dim], wk/wv [q_dim, d_in],
       wout [width, n_queries*q_dim], bout [width] */
    const uint16_t *q, *wk, *wv, *wout, *bout;
} jnx_head;

/* Per-slot fp32 gradient buffers, same shapes as the parameters.  w1,
 * w2 / wout and q (parameters), and the gradients' w2 / wout, wk and wv,
 * must be 16-byte aligned, and the heads of one group share d_in
 * (JNX_ERR_INVALID_ARG / JNX_ERR_UNSUPPORTED otherwise). */
typedef struct {
    float *w1, *b1, *w2, *b2;
    float *q, *wk, *wv, *wout, *bout;
} jnx_head_grads;

/* Workspace bytes jnx_heads_forward / jnx_heads_backward need. */
size_t jnx_heads_workspace_bytes(const jnx_head* heads, int32_t n_tenants, const jnx_group* g);

/* Each group slot's head on that tenant's samples only.  heads[] is a HOST
 * array indexed by tenant.  Writes preds at each sample's target offset
 * (arrival layout, fp32) and loss[tenant] = mean squared error over the
 * tenant's samples and outputs, for the tenants in the group only.  The
 * activations the backward needs are kept in `workspace`.  targets and loss
 * may both be NULL (inference: predictions only; a jnx_heads_backward then
 * needs a forward with targets first). */
jnx_status jnx_heads_forward(const jnx_head* heads, int32_t n_tenants, const jnx_group* g,
                             const float* pooled, const uint16_t* hidden,
                             const float* targets, float* preds, float* loss,
                             void* workspace, size_t ws_bytes, void* stream);

/* Gradients of each group tenant's loss w.r.t. that tenant's head
 * parameters, written (overwritten, fp32) into grads[tenant] only; slots of
 * tenants outside the group are not touched.  Must follow jnx_heads_forward
 * on the same stream with the same group, features, targets and workspace:
 * it reads the activations that call stored there.  No feature gradient is
 * produced (the backbone is frozen). */
jnx_status jnx_heads_backward(const jnx_head* heads, int32_t n_tenants, const jnx_group* g,
                              const float* pooled, const uint16_t* hidden,
                              const float* targets, const jnx_head_grads* grads,
                              void* workspace, size_t ws_bytes, void* stream);

/* Same, but adds the gradients into grads[tenant] (gradient accumulation
 * over successive groups before an optimizer step) instead of overwriting. */
jnx_status jnx_heads_backward_accumulate(const jnx_head* heads, int32_t n_tenants,
                                         const jnx_group* g, const float* pooled,
                                         const uint16_t* hidden, const float* targets,
                                         const jnx_head_grads* grads, void* workspace,
                                         size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Tenant-private optimizer step
 * ------------------------------------------------------------------------ */

/* One tenant's head optimizer state (App. A, "Actor Consumption and Version
 * Consistency": only that tenant's optimizer runs on its microbatch and only
 * its policy version increments; nothing is shared across tenants).  Device
 * fp32 arrays with the shapes of the head's parameters, indexed in the order
 * w1, b1, w2, b2, q, wk, wv, wout, bout (NULL for the parameters the head's
 * kind does not have): the master copy the updates act on, and AdamW's first
 * and second moments (zero before the first step).  step and version are
 * host counters that jnx_heads_adamw increments. */
typedef struct {
    float* master[9];
    float* m[9];
    float* v[9];
    int32_t step;     /* AdamW steps taken */
    int32_t version;  /* policy version */
} jnx_head_opt;

typedef struct {
    float lr, beta1, beta2, eps, weight_decay;
} jnx_adamw;

/* One AdamW step (decoupled weight decay) on the head of every tenant in the
 * group, from its fp32 gradients: per element, with t = opt[tenant].step + 1,
 *   m <- b1 m + (1 - b1) g,  v <- b2 v + (1 - b2) g^2,
 *   master <- master - lr ((m / (1 - b1^t)) / (sqrt(v / (1 - b2^t)) + eps)
 *                          + weight_decay master),
 * then the head's bf16 parameter (written in place through the jnx_head
 * pointers) = master rounded to nearest even; opt[tenant].step and .version
 * increment.  fp32 arithmetic.  Tenants outside the group are not touched.
 * heads[] and opt[] are HOST arrays indexed by tenant.  Errors:
 * JNX_ERR_INVALID_ARG (null state for a parameter the head has, lr < 0,
 * b1 or b2 outside [0, 1), eps < 0, weight_decay < 0); nothing is written
 * on error. */
jnx_status jnx_heads_adamw(const jnx_head* heads, const jnx_head_grads* grads,
                           jnx_head_opt* opt, int32_t n_tenants, const jnx_group* g,
                           const jnx_adamw* hp, void* stream);

/* The heads backward with each group tenant's AdamW step fused into it
 * (App. A "Actor Consumption and Version Consistency": a microbatch steps
 * only its own tenant's optimizer and policy version; nothing is shared or
 * averaged across tenants).  The result equals jnx_heads_backward (or, with
 * accumulate != 0, jnx_heads_backward_accumulate) followed by
 * jnx_heads_adamw, but no gradient is stored: each gradient element goes
 * straight into its parameter's update, which saves writing and re-reading
 * the fp32 gradients.  accumulate != 0 adds grads[tenant] (the earlier
 * microbatches' sum, read, not written) to this backward's gradient before
 * the step; accumulate == 0 never touches grads (may be NULL).  d_hidden
 * (optional, [n_tokens, d] fp32, as jnx_heads_backward_input) receives the
 * gradient at the final normed rows, formed from the parameters before
 * their update.  Every parameter is read before it is updated.  On success
 * opt[tenant].step and .version are incremented for the group's tenants.
 * Errors as jnx_heads_backward and jnx_heads_adamw (null or misaligned
 * optimizer state: JNX_ERR_INVALID_ARG before any launch).  A capturing
 * stream is accepted (nothing is uploaded from host memory). */
jnx_status jnx_heads_backward_adamw(const jnx_head* heads, int32_t n_tenants,
                                    const jnx_group* g, const float* pooled,
                                    const uint16_t* hidden, const float* targets,
                                    const jnx_head_grads* grads, int32_t accumulate,
                                    jnx_head_opt* opt, const jnx_adamw* hp, float* d_hidden,
                                    void* workspace, size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Trainable per-tenant adapters: the LoRA backward through the frozen backbone
 *
 * A tenant's trainable module may be a lightweight adapter over the fixed
 * base (§3.1); its loss, gradients and optimizer state stay its own (§5.2,
 * App. A).  With the backbone's LoRA adapters (lora_rank 16), one grouped
 * step gives every group tenant the gradient of its own loss with respect
 * to its own adapters:
 *   jnx_backbone_forward_train   forward, keeping each block's residual input
 *   jnx_heads_forward            per-tenant heads and losses
 *   jnx_heads_backward_input     head gradients + dloss/d(final normed rows)
 *   jnx_backbone_backward_lora   adapter gradients of every layer
 * ------------------------------------------------------------------------ */

/* Bytes of the buffer jnx_backbone_forward_train keeps: fp32
 * [n_layers + 1, n_tokens, d_model]. */
size_t jnx_backbone_saved_bytes(const jnx_backbone* bb, int32_t n_tokens);

/* jnx_backbone_forward that also writes saved[l] = the fp32 residual stream
 * entering block l (l < n_layers) and saved[n_layers] = the one entering
 * the final RMSNorm. */
jnx_status jnx_backbone_forward_train(const jnx_backbone* bb, const jnx_group* g,
                                      const uint16_t* vision, int64_t n_vision_rows,
                                      const int32_t* text_ids, int64_t n_text,
                                      float* pooled, uint16_t* hidden, float* saved,
                                      void* workspace, size_t ws_bytes, void* stream);

/* jnx_heads_backward, and also d_hidden [n_tokens, d] fp32 = the gradient
 * of each row's tenant loss with respect to that row's final normed
 * hidden: (dz W1) / L_s on every row of an MLP-head sample (the feature is
 * the mean of the rows), dk W_k + dv W_v on a query-head row.  Every row of
 * the group is written. */
jnx_status jnx_heads_backward_input(const jnx_head* heads, int32_t n_tenants,
                                    const jnx_group* g, const float* pooled,
                                    const uint16_t* hidden, const float* targets,
                                    const jnx_head_grads* grads, float* d_hidden,
                                    void* workspace, size_t ws_bytes, void* stream);

/* Transposed copies of one block's frozen weights (device bf16), read by
 * the backward's input-gradient GEMMs; jnx_transpose builds them once.
 *   w_qkv_t  [d, (H + 2 Hkv) hd] = w_qkv^T
 *   w_o_t    [H hd, d]           = w_o^T
 *   w_gu_t   [d, 2 F]            = w_gu^T (columns in w_gu's packed row order)
 *   w_down_t [F, d]              = w_down^T */
typedef struct {
    const uint16_t* w_qkv_t;
    const uint16_t* w_o_t;
    const uint16_t* w_gu_t;
    const uint16_t* w_down_t;
} jnx_layer_t;

/* One block's adapter gradients (device fp32), the shapes of the adapters:
 * a_* [n_tenants, r, in], b_* [n_tenants, out, r]. */
typedef struct {
    float *a_q, *b_q, *a_k, *b_k, *a_v, *b_v, *a_o, *b_o;
} jnx_lora_grads;

/* dst [batch][cols][rows] = src [batch][rows][cols] (bf16, not in place). */
jnx_status jnx_transpose(const uint16_t* src, int32_t batch, int32_t rows, int32_t cols,
                         uint16_t* dst, void* stream);

/* Workspace bytes jnx_backbone_backward_lora needs for n_tokens rows. */
size_t jnx_backbone_backward_workspace_bytes(const jnx_backbone* bb, int32_t n_tokens);

/* The gradient of each group tenant's loss with respect to its own LoRA
 * adapters in every block, written (accumulate == 0) or added into the
 * tenant's slice of grads[l] (HOST array [n_layers]); slices of tenants
 * outside the group are not touched.  saved: what jnx_backbone_forward_train
 * kept for this group; d_hidden [n_tokens, d] fp32: dloss/d(final normed
 * rows) (jnx_heads_backward_input).  layers_t: HOST array [n_layers] of the
 * transposed weights.  Each block is recomputed from its saved input.
 * Errors: JNX_ERR_INVALID_ARG (no rank-16 adapters, null buffer, a group
 * tenant without an adapter), JNX_ERR_UNSUPPORTED (widths not multiples of
 * 256, more than 256 group tenants), JNX_ERR_WORKSPACE. */
jnx_status jnx_backbone_backward_lora(const jnx_backbone* bb, const jnx_layer_t* layers_t,
                                      const jnx_group* g, const float* saved,
                                      const float* d_hidden, const jnx_lora_grads* grads,
                                      int32_t accumulate, void* workspace, size_t ws_bytes,
                                      void* stream);

/* ------------------------------------------------------------------------
 * Flow-matching action expert (a DiT head) as the tenant's private module
 *
 * §3.1 names diffusion / flow-matching action experts among the action
 * modules; §5.2 trains QwenGR00T's GR00T-style flow-matching head (and
 * pi-0.5's) as the tenant-private module over the shared VLM.  The paper
 * gives no equations; the expert here (per sample s of tenant t, context
 * X = the sample's final normed backbone rows [L, d]):
 *   x = tau a + (1 - tau) eps  (a: target chunk [C, D], eps: noise, tau in [0, 1]
 *                               drawn by the caller), u = a - eps
 *   phi = T2 SiLU(T1 s(tau) + tb1) + tb2, s(tau) = [sin(1000 tau w_i) | cos(...)],
 *         w_i = 10000^(-i / (dm/2))
 *   h = x W_in^T + b_in + pos + phi                                     [C, dm]
 *   per block: q|k_a|v_a = n(h) W_qkv^T, k_c|v_c = X W_kvc^T,
 *              h += MHA(q; [k_c; k_a], [v_c; v_a]) W_o^T   (heads of 64)
 *              h += W_d (SiLU(n(h) W_g^T) * (n(h) W_u^T))
 *   v = n(h) W_out^T + b_out,  n(h) = h / sqrt(mean(h^2) + 1e-6)
 *   loss_t = mean over the tenant's samples and chunk elements of (v - u)^2
 * Every tenant of a call has the same dimensions; parameters are stacked
 * over tenants (bf16, tenant t's slice at t times the per-tenant size).
 * ------------------------------------------------------------------------ */

typedef struct {
    const uint16_t* w_qkv;  /* [T, 3 dm, dm]: rows of W_q, W_k (action), W_v (action) */
    const uint16_t* w_kvc;  /* [T, 2 dm, d]: rows of W_k, W_v over the context */
    const uint16_t* w_o;    /* [T, dm, dm] */
    const uint16_t* w_gu;   /* [T, 2 F, dm]: W_g, W_u in jnx_pack_gate_up's packed order */
    const uint16_t* w_d;    /* [T, dm, F] */
} jnx_flow_block;

typedef struct {
    int32_t d_model;     /* dm: 256, 512 or 1024 (heads of 64) */
    int32_t d_ff;        /* F: a multiple of 128 */
    int32_t n_blocks;
    int32_t chunk;       /* C: 1..64 action steps */
    int32_t action_dim;  /* D: 1..64 */
    int32_t d_in;        /* the backbone width d (a multiple of 128) */
    int32_t n_tenants;   /* T: tenants the stacked arrays hold */
    const uint16_t* w_in;   /* [T, dm, D] */
    const uint16_t* b_in;   /* [T, dm] */
    const uint16_t* pos;    /* [T, C, dm] */
    const uint16_t* t1;     /* [T, dm, dm] */
    const uint16_t* tb1;    /* [T, dm] */
    const uint16_t* t2;     /* [T, dm, dm] */
    const uint16_t* tb2;    /* [T, dm] */
    const uint16_t* w_out;  /* [T, D, dm] */
    const uint16_t* b_out;  /* [T, D] */
    const jnx_flow_block* blocks;  /* HOST array [n_blocks] */
} jnx_flow_head;

/* Gradients (device fp32), the shapes of the stacked parameters. */
typedef struct {
    float *w_qkv, *w_kvc, *w_o, *w_gu, *w_d;
} jnx_flow_block_grads;

typedef struct {
    float *w_in, *b_in, *pos, *t1, *tb1, *t2, *tb2, *w_out, *b_out;
    const jnx_flow_block_grads* blocks;  /* HOST array [n_blocks] */
} jnx_flow_grads;

/* Workspace bytes of jnx_flow_forward / jnx_flow_backward / jnx_flow_sample.
 * The workspace must be 256-byte aligned and the t1, t2 and w_out weights
 * 16-byte aligned (JNX_ERR_INVALID_ARG otherwise). */
size_t jnx_flow_workspace_bytes(const jnx_flow_head* fh, const jnx_group* g);

/* Training forward of every group tenant's expert over its samples.
 * hidden [n_tokens, d] bf16: the backbone's final normed rows.  actions,
 * noise [n_samples, C, D] fp32 and tau [n_samples] fp32 in the group's
 * packed sample order; velocity [n_samples, C, D] fp32 (out);
 * loss[tenant] fp32 for the group's tenants.  Keeps the activations the
 * backward needs in `workspace`.  Every group tenant must be < n_tenants. */
jnx_status jnx_flow_forward(const jnx_flow_head* fh, const jnx_group* g, const uint16_t* hidden,
                            const float* actions, const float* noise, const float* tau,
                            float* velocity, float* loss, void* workspace, size_t ws_bytes,
                            void* stream);

/* Gradients of each group tenant's loss with respect to its own expert
 * parameters, written (accumulate == 0) or added into the tenant's slices
 * of `grads`; other tenants' slices are not touched.  Must follow
 * jnx_flow_forward with the same group, hidden rows and workspace. */
jnx_status jnx_flow_backward(const jnx_flow_head* fh, const jnx_group* g, const uint16_t* hidden,
                             const jnx_flow_grads* grads, int32_t accumulate, void* workspace,
                             size_t ws_bytes, void* stream);

/* Inference: from x = noise at tau = 0, n_steps Euler steps of
 * x += v(x, tau) / n_steps up to tau = 1 (the context's K/V projections are
 * computed once and reused by every step).  actions [n_samples, C, D] fp32
 * (out), packed sample order. */
jnx_status jnx_flow_sample(const jnx_flow_head* fh, const jnx_group* g, const uint16_t* hidden,
                           const float* noise, int32_t n_steps, float* actions, void* workspace,
                           size_t ws_bytes, void* stream);

/* ------------------------------------------------------------------------
 * Tenant-private optimizer step on any trainable tensors
 * ------------------------------------------------------------------------ */

/* One tenant-private parameter tensor (device): its bf16 value the kernels
 * read (written in place), fp32 master copy, AdamW moments (zero before the
 * first step), fp32 gradient, element count, and the number of steps this
 * tensor has taken (a host counter the call increments).  A LoRA adapter's
 * or a flow expert's slice of one tenant is one such tensor. */
typedef struct {
    uint16_t* param;
    float* master;
    float* m;
    float* v;
    const float* grad;
    int64_t n;
    int32_t* step;
} jnx_adam_tensor;

/* One AdamW step (the update of jnx_heads_adamw) on each tensor, with
 * t = *step + 1 for that tensor; then each *step increments.  Errors:
 * JNX_ERR_INVALID_ARG (null buffer, n < 0, hyperparameters as for
 * jnx_heads_adamw); nothing is written on error. */
jnx_status jnx_adamw_tensors(const jnx_adam_tensor* tensors, int32_t n_tensors,
                             const jnx_adamw* hp, void* stream);

/* ------------------------------------------------------------------------
 * Status and helpers
 * ------------------------------------------------------------------------ */

/* Synchronise `stream`, read and clear the device status word at the start
 * of `workspace`; returns JNX_OK or the first error a kernel recorded. */
jnx_status jnx_check_status(void* workspace, void* stream);

/* Build the interleaved w_gu layout from W_g [F, d] and W_u [F, d]
 * (F a multiple of 128).  out [2F, d]. */
jnx_status jnx_pack_gate_up(const uint16_t* w_gate, const uint16_t* w_up, int32_t F, int32_t d,
                            uint16_t* out, void* stream);


/* ------------------------------------------------------------------------
 * Kernel tracing (host thread local)
 * ------------------------------------------------------------------------ */

/* Kernel ids reported by the tracer. */
#define JNX_K_PACK 1       /* work = HBM bytes */
#define JNX_K_RMSNORM 2    /* work = HBM bytes */
#define JNX_K_GEMM_QKV 3   /* work = FLOPs */
#define JNX_K_ATTN 4       /* work = FLOPs (within-sample only) */
#define JNX_K_GEMM_O 5     /* work = FLOPs */
#define JNX_K_GEMM_GU 6    /* work = FLOPs */
#define JNX_K_GEMM_DOWN 7  /* work = FLOPs */
#define JNX_K_POOL 8       /* work = HBM bytes */
#define JNX_K_ROPE_TABLE 9 /* work = bytes written */
#define JNX_K_HEADS_FWD 10 /* work = FLOPs */
#define JNX_K_HEADS_BWD 11 /* work = FLOPs */
#define JNX_K_GEMM 12      /* jnx_op_gemm; work = FLOPs */
#define JNX_K_LORA 13      /* LoRA row tenants / down-projections; work = FLOPs */
#define JNX_K_ADAMW 14     /* tenant-private head optimizer step; work = HBM bytes */
#define JNX_K_GEMM_BWD 15  /* input-gradient GEMMs of the adapter backward; work = FLOPs */
#define JNX_K_ATTN_BWD 16  /* attention backward; work = FLOPs of its five products */
#define JNX_K_NORM_BWD 17  /* RMSNorm backward, attention-backward prologue; work = HBM bytes */
#define JNX_K_LORA_BWD 18  /* adapter gradients and up-projections; work = FLOPs */
#define JNX_K_FLOW_GEMM 19 /* flow expert: segmented projections; work = FLOPs */
#define JNX_K_FLOW_ATTN 20 /* flow expert: attention forward / backward; work = FLOPs */
#define JNX_K_FLOW_MISC 21 /* flow expert: time / embedding / output / norms / reductions */
#define JNX_K_FLOW_WGRAD 22 /* flow expert: weight gradients; work = FLOPs */

/* While enabled on the calling thread, each kernel launch of the library is
 * bracketed by two CUDA events on its stream (up to `capacity` launches are
 * kept; later ones are only counted).  Enabling resets the record. */
jnx_status jnx_trace_enable(int32_t capacity);
jnx_status jnx_trace_disable(void);
/* Launches seen since the last enable (including those past capacity). */
int32_t jnx_trace_count(void);
/* Waits for the recorded events and returns, per recorded launch, its kernel
 * id, its duration in ms and its algorithmic work; *n_out = entries written. */
jnx_status jnx_trace_read(int32_t* kinds, float* ms, double* work, int32_t cap, int32_t* n_out);

#ifdef __cplusplus
}
#endif

#endif /* JNX_H */
