// jnx_group_plan: FIFO-compatible prefix collection and canonical packing.
//
// App. A ("Inference Queue Composition"): requests are examined in arrival
// order; the scheduler keeps the largest prefix that is compatible at the
// shared frozen-prefix boundary and fits the batch limits; canonicalisation
// produces one physical encoder batch and the slices that route features
// back.  §4.3: the canonical VLAFeature is where tenants' samples are
// concatenated.  Packing is varlen (no padding) so grouped results equal
// per-sample results.
#include <cmath>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include "jnx_host.h"

namespace jnx {

static thread_local std::string g_last_error;

jnx_status fail(jnx_status code, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return code;
}

void clear_error() { g_last_error.clear(); }

static bool same_prefix(const jnx_schema& a, const jnx_schema& b) {
    return a.backbone_id == b.backbone_id && a.d_model == b.d_model &&
           a.vision_tokens == b.vision_tokens && a.embed_dtype == b.embed_dtype &&
           a.vocab_id == b.vocab_id && a.rope_id == b.rope_id;
}

static int64_t sample_len(const jnx_schema& sc, const jnx_sample& s) {
    return (int64_t)s.n_img * sc.vision_tokens + s.text_len;
}

// Every request of a queue well formed (tenant, schema, sample shapes and
// offsets within int32).
static jnx_status validate_requests(const jnx_schema* schemas, int32_t n_schemas,
                                    const jnx_request* reqs, int32_t n_reqs, int32_t n_tenants) {
    for (int32_t i = 0; i < n_reqs; ++i) {
        const jnx_request& r = reqs[i];
        if (r.tenant < 0 || r.tenant >= n_tenants)
            return fail(JNX_ERR_INVALID_ARG, "request %d: tenant %d outside [0, %d)", i, r.tenant,
                        n_tenants);
        if (r.schema < 0 || r.schema >= n_schemas)
            return fail(JNX_ERR_INVALID_ARG, "request %d: schema %d out of range", i, r.schema);
        if (r.n_samples < 1 || !r.samples)
            return fail(JNX_ERR_INVALID_ARG, "request %d: no samples", i);
        const jnx_schema& sc = schemas[r.schema];
        if (sc.vision_tokens < 0 || sc.action_width < 0 || sc.max_images < 0)
            return fail(JNX_ERR_INVALID_ARG, "schema %d: negative field", r.schema);
        for (int32_t j = 0; j < r.n_samples; ++j) {
            const jnx_sample& s = r.samples[j];
            if (s.n_img < 0 || s.n_img > sc.max_images || s.text_len < 0)
                return fail(JNX_ERR_INVALID_ARG, "request %d sample %d: bad shape", i, j);
            if (sample_len(sc, s) < 1)
                return fail(JNX_ERR_INVALID_ARG, "request %d sample %d: empty sample", i, j);
            const int64_t vr_end = s.vision_row + (int64_t)s.n_img * sc.vision_tokens;
            const int64_t tp_end = s.text_pos + s.text_len;
            const int64_t tg_end = s.target_off + sc.action_width;
            if (s.vision_row < 0 || s.text_pos < 0 || s.target_off < 0)
                return fail(JNX_ERR_INVALID_ARG, "request %d sample %d: negative offset", i, j);
            if (vr_end > INT32_MAX || tp_end >= INT32_MAX || tg_end > INT32_MAX ||
                sample_len(sc, s) > INT32_MAX)
                return fail(JNX_ERR_OVERFLOW, "request %d sample %d: offset beyond int32", i, j);
        }
    }
    return JNX_OK;
}

}  // namespace jnx

using namespace jnx;

extern "C" const char* jnx_last_error(void) { return g_last_error.c_str(); }

extern "C" int32_t jnx_version(void) { return 1; }

extern "C" jnx_status jnx_group_plan(const jnx_schema* schemas, int32_t n_schemas,
                                     const jnx_request* reqs, int32_t n_reqs, int32_t n_tenants,
                                     const jnx_limits* lim, jnx_plan* out) {
    clear_error();
    if (!out || !lim || n_reqs < 0 || n_tenants < 0 || (n_reqs > 0 && (!reqs || !schemas)))
        return fail(JNX_ERR_INVALID_ARG, "jnx_group_plan: null argument or negative count");

    // Validate every request in the queue before deciding anything.
    if (jnx_status st = validate_requests(schemas, n_schemas, reqs, n_reqs, n_tenants)) return st;

    // Largest FIFO-compatible prefix under the limits (whole requests).
    int32_t k = 0;
    int64_t n_s = 0, n_t = 0;
    if (n_reqs > 0) {
        const jnx_schema& key = schemas[reqs[0].schema];
        for (int32_t i = 0; i < n_reqs; ++i) {
            const jnx_request& r = reqs[i];
            const jnx_schema& sc = schemas[r.schema];
            if (!same_prefix(sc, key)) break;
            int64_t rt = 0;
            for (int32_t j = 0; j < r.n_samples; ++j) rt += sample_len(sc, r.samples[j]);
            if (k > 0 && (n_s + r.n_samples > lim->max_samples || n_t + rt > lim->max_tokens))
                break;
            n_s += r.n_samples;
            n_t += rt;
            ++k;
        }
    }
    if (n_t > INT32_MAX) return fail(JNX_ERR_OVERFLOW, "packed batch over int32 tokens");

    // Group slots in order of first appearance.
    std::vector<int32_t> slot_tenant;
    std::vector<int32_t> slot_of(n_tenants, -1);
    for (int32_t i = 0; i < k; ++i) {
        const int32_t t = reqs[i].tenant;
        if (slot_of[t] < 0) {
            slot_of[t] = (int32_t)slot_tenant.size();
            slot_tenant.push_back(t);
        }
    }
    const int32_t G = (int32_t)slot_tenant.size();

    out->n_requests = k;
    out->n_samples = (int32_t)n_s;
    out->n_tokens = (int32_t)n_t;
    out->n_slots = G;
    out->max_seqlen = 0;
    if (n_s > out->cap_samples || n_t > out->cap_tokens || G > out->cap_slots)
        return fail(JNX_ERR_CAPACITY, "plan needs %lld samples, %lld tokens, %d slots",
                    (long long)n_s, (long long)n_t, G);
    if (!out->cu_seqlens || !out->sample_slot || !out->sample_req || !out->sample_target ||
        !out->sample_width || !out->seg_offsets || !out->slot_tenant ||
        (n_t > 0 && (!out->gather_src || !out->pos_ids)))
        return fail(JNX_ERR_INVALID_ARG, "jnx_group_plan: null output array");

    // Requests of each slot in FIFO order (a bucket list keeps this O(k)).
    std::vector<std::vector<int32_t>> reqs_of(G);
    for (int32_t i = 0; i < k; ++i) reqs_of[slot_of[reqs[i].tenant]].push_back(i);

    int32_t S = 0, tok = 0, maxlen = 0;
    out->cu_seqlens[0] = 0;
    out->seg_offsets[0] = 0;
    for (int32_t g = 0; g < G; ++g) {
        out->slot_tenant[g] = slot_tenant[g];
        for (int32_t ri : reqs_of[g]) {
            const jnx_request& r = reqs[ri];
            const jnx_schema& sc = schemas[r.schema];
            for (int32_t j = 0; j < r.n_samples; ++j) {
                const jnx_sample& s = r.samples[j];
                const int32_t nv = s.n_img * sc.vision_tokens;
                const int32_t L = nv + s.text_len;
                for (int32_t q = 0; q < nv; ++q) {
                    out->gather_src[tok + q] = (int32_t)(s.vision_row + q);
                    out->pos_ids[tok + q] = q;
                }
                for (int32_t q = 0; q < s.text_len; ++q) {
                    out->gather_src[tok + nv + q] = -(int32_t)(s.text_pos + q) - 1;
                    out->pos_ids[tok + nv + q] = nv + q;
                }
                tok += L;
                if (L > maxlen) maxlen = L;
                out->cu_seqlens[S + 1] = tok;
                out->sample_slot[S] = g;
                out->sample_req[S] = ri;
                out->sample_target[S] = (int32_t)s.target_off;
                out->sample_width[S] = sc.action_width;
                ++S;
            }
        }
        out->seg_offsets[g + 1] = S;
    }
    out->max_seqlen = maxlen;
    return JNX_OK;
}

// jnx_sched_poll: the inference scheduler's decision at time `now`.
//
// §4.3: the inference service keeps a maximum waiting time T and a target
// batch size B, builds a batch from requests in FIFO order and starts it
// when the waiting time reaches T or the batch size reaches B.  App. A: the
// batch is the largest FIFO-compatible prefix the limits allow.  The batch
// is collected as jnx_group_plan collects it (compatibility with the oldest
// request, whole requests, the oldest always taken); it also fires when the
// batch cannot grow because the next compatible request does not fit.  The
// skip-ahead mode passes over incompatible requests, which stay queued.
extern "C" jnx_status jnx_sched_poll(const jnx_schema* schemas, int32_t n_schemas,
                                     const jnx_request* reqs, const double* arrival,
                                     int32_t n_reqs, int32_t n_tenants, double now,
                                     const jnx_sched_policy* pol, int32_t* take, int32_t* n_take,
                                     double* wake) {
    clear_error();
    if (!pol || !n_take || !wake || n_reqs < 0 || n_tenants < 0 ||
        (n_reqs > 0 && (!reqs || !schemas || !arrival || !take)))
        return fail(JNX_ERR_INVALID_ARG, "jnx_sched_poll: null argument or negative count");
    if (pol->batch_samples < 1 || pol->max_tokens < 1 || !(pol->timeout >= 0.0) ||
        (pol->skip_ahead != 0 && pol->skip_ahead != 1))
        return fail(JNX_ERR_INVALID_ARG, "jnx_sched_poll: bad policy");
    if (jnx_status st = validate_requests(schemas, n_schemas, reqs, n_reqs, n_tenants)) return st;
    *n_take = 0;
    if (n_reqs == 0) {
        *wake = HUGE_VAL;
        return JNX_OK;
    }
    const jnx_schema& key = schemas[reqs[0].schema];
    int32_t k = 0;
    int64_t n_s = 0, n_t = 0;
    bool full = false;
    for (int32_t i = 0; i < n_reqs; ++i) {
        const jnx_request& r = reqs[i];
        const jnx_schema& sc = schemas[r.schema];
        if (!same_prefix(sc, key)) {
            if (pol->skip_ahead) continue;
            break;
        }
        int64_t rt = 0;
        for (int32_t j = 0; j < r.n_samples; ++j) rt += sample_len(sc, r.samples[j]);
        if (k > 0 && (n_s + r.n_samples > pol->batch_samples || n_t + rt > pol->max_tokens)) {
            full = true;
            break;
        }
        take[k++] = i;
        n_s += r.n_samples;
        n_t += rt;
    }
    if (n_s >= pol->batch_samples || full || now - arrival[0] >= pol->timeout) {
        *n_take = k;
        *wake = now;
    } else {
        *wake = arrival[0] + pol->timeout;
    }
    return JNX_OK;
}
