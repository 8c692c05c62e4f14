"""ctypes binding of libjnx.so: the C ABI of include/jnx.h and include/jnx_ops.h
under the same names.  Argument marshalling only — every step of the path
runs in the library's CUDA kernels; nothing here computes.

The library must be built (``paper_2607_16074_gb300.build``); importing this
module does not fall back to anything if it is missing: ``lib()`` raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional, Sequence

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libjnx.so")

JNX_OK = 0
ERRORS = {-1: "INVALID_ARG", -3: "CAPACITY", -5: "OVERFLOW", -6: "CUDA", -7: "DEVICE_BOUNDS",
          -8: "TIMEOUT", -9: "UNSUPPORTED", -10: "WORKSPACE"}
JNX_ERR_INVALID_ARG, JNX_ERR_CAPACITY, JNX_ERR_OVERFLOW = -1, -3, -5
JNX_ERR_CUDA, JNX_ERR_DEVICE_BOUNDS, JNX_ERR_TIMEOUT = -6, -7, -8
JNX_ERR_UNSUPPORTED, JNX_ERR_WORKSPACE = -9, -10
JNX_GLU_SWIGLU, JNX_GLU_GEGLU_TANH = 0, 1
JNX_HEAD_MLP, JNX_HEAD_XATTN = 0, 1
JNX_EPI_BF16, JNX_EPI_F32, JNX_EPI_RESID, JNX_EPI_GLU, JNX_EPI_ROPE = 0, 1, 2, 3, 4
JNX_EPI_GLU_SAVE = 6
JNX_NOALLOC_MAX_ROPE_ENTRIES = 1 << 19


class JnxError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"jnx error {code} ({ERRORS.get(code, '?')}): {msg}")
        self.code = code


P32 = C.POINTER(C.c_int32)
PU16 = C.c_void_p  # bf16 arrays are passed as raw addresses


class jnx_schema(C.Structure):
    _fields_ = [("backbone_id", C.c_int32), ("d_model", C.c_int32), ("vision_tokens", C.c_int32),
                ("embed_dtype", C.c_int32), ("vocab_id", C.c_int32), ("rope_id", C.c_int32),
                ("max_images", C.c_int32), ("action_width", C.c_int32)]


class jnx_sample(C.Structure):
    _fields_ = [("n_img", C.c_int32), ("text_len", C.c_int32), ("vision_row", C.c_int64),
                ("text_pos", C.c_int64), ("target_off", C.c_int64)]


class jnx_request(C.Structure):
    _fields_ = [("tenant", C.c_int32), ("schema", C.c_int32), ("n_samples", C.c_int32),
                ("reserved", C.c_int32), ("samples", C.POINTER(jnx_sample))]


class jnx_limits(C.Structure):
    _fields_ = [("max_samples", C.c_int32), ("max_tokens", C.c_int32)]


class jnx_plan(C.Structure):
    _fields_ = [("cap_samples", C.c_int32), ("cap_tokens", C.c_int32), ("cap_slots", C.c_int32),
                ("n_requests", C.c_int32), ("n_samples", C.c_int32), ("n_tokens", C.c_int32),
                ("n_slots", C.c_int32), ("max_seqlen", C.c_int32),
                ("cu_seqlens", P32), ("sample_slot", P32), ("sample_req", P32),
                ("sample_target", P32), ("sample_width", P32), ("seg_offsets", P32),
                ("slot_tenant", P32), ("gather_src", P32), ("pos_ids", P32)]


class jnx_sched_policy(C.Structure):
    _fields_ = [("timeout", C.c_double), ("batch_samples", C.c_int32), ("max_tokens", C.c_int32),
                ("skip_ahead", C.c_int32), ("reserved", C.c_int32)]


class jnx_group(C.Structure):
    _fields_ = [("n_samples", C.c_int32), ("n_tokens", C.c_int32), ("n_slots", C.c_int32),
                ("max_seqlen", C.c_int32),
                ("cu_seqlens", C.c_void_p), ("sample_slot", C.c_void_p),
                ("sample_target", C.c_void_p), ("seg_offsets", C.c_void_p),
                ("gather_src", C.c_void_p), ("pos_ids", C.c_void_p),
                ("h_cu_seqlens", P32), ("h_seg_offsets", P32), ("h_slot_tenant", P32),
                ("attn_items", C.c_void_p), ("n_attn_items", C.c_int32)]


class jnx_layer(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in (
        "attn_norm", "w_qkv", "w_o", "ffn_norm", "w_gu", "w_down",
        "lora_a_q", "lora_b_q", "lora_a_k", "lora_b_k", "lora_a_v", "lora_b_v",
        "lora_a_o", "lora_b_o")]


class jnx_backbone(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("d_model", C.c_int32), ("n_heads", C.c_int32),
                ("n_kv_heads", C.c_int32), ("head_dim", C.c_int32), ("d_ff", C.c_int32),
                ("glu", C.c_int32), ("lora_rank", C.c_int32), ("n_tenants", C.c_int32),
                ("vocab", C.c_int32), ("vision_tokens", C.c_int32), ("eps", C.c_float),
                ("rope_theta", C.c_float), ("text_table", C.c_void_p), ("final_norm", C.c_void_p),
                ("layers", C.POINTER(jnx_layer))]


class jnx_head(C.Structure):
    _fields_ = [("kind", C.c_int32), ("d_in", C.c_int32), ("d_hidden", C.c_int32),
                ("n_queries", C.c_int32), ("q_dim", C.c_int32), ("width", C.c_int32)] + \
               [(n, C.c_void_p) for n in ("w1", "b1", "w2", "b2", "q", "wk", "wv", "wout", "bout")]


class jnx_head_grads(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("w1", "b1", "w2", "b2", "q", "wk", "wv", "wout",
                                          "bout")]


HEAD_PARAMS = ("w1", "b1", "w2", "b2", "q", "wk", "wv", "wout", "bout")


class jnx_head_opt(C.Structure):
    _fields_ = [("master", C.c_void_p * 9), ("m", C.c_void_p * 9), ("v", C.c_void_p * 9),
                ("step", C.c_int32), ("version", C.c_int32)]


class jnx_adamw(C.Structure):
    _fields_ = [("lr", C.c_float), ("beta1", C.c_float), ("beta2", C.c_float),
                ("eps", C.c_float), ("weight_decay", C.c_float)]


class jnx_layer_t(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("w_qkv_t", "w_o_t", "w_gu_t", "w_down_t")]


LORA_GRADS = ("a_q", "b_q", "a_k", "b_k", "a_v", "b_v", "a_o", "b_o")


class jnx_lora_grads(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in LORA_GRADS]


class jnx_flow_block(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in ("w_qkv", "w_kvc", "w_o", "w_gu", "w_d")]


class jnx_flow_head(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("d_model", "d_ff", "n_blocks", "chunk", "action_dim",
                                         "d_in", "n_tenants")] + \
               [(n, C.c_void_p) for n in ("w_in", "b_in", "pos", "t1", "tb1", "t2", "tb2",
                                          "w_out", "b_out")] + \
               [("blocks", C.POINTER(jnx_flow_block))]


FLOW_PARAMS = ("w_in", "b_in", "pos", "t1", "tb1", "t2", "tb2", "w_out", "b_out")
FLOW_BLOCK_PARAMS = ("w_qkv", "w_kvc", "w_o", "w_gu", "w_d")


class jnx_flow_block_grads(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in FLOW_BLOCK_PARAMS]


class jnx_flow_grads(C.Structure):
    _fields_ = [(n, C.c_void_p) for n in FLOW_PARAMS] + \
               [("blocks", C.POINTER(jnx_flow_block_grads))]


class jnx_adam_tensor(C.Structure):
    _fields_ = [("param", C.c_void_p), ("master", C.c_void_p), ("m", C.c_void_p),
                ("v", C.c_void_p), ("grad", C.c_void_p), ("n", C.c_int64),
                ("step", C.POINTER(C.c_int32))]


_LIB: Optional[C.CDLL] = None

EXPORTS = ("jnx_last_error", "jnx_version", "jnx_group_plan", "jnx_group_attn_items",
           "jnx_backbone_workspace_bytes",
           "jnx_backbone_forward", "jnx_heads_workspace_bytes", "jnx_heads_forward",
           "jnx_heads_backward", "jnx_check_status", "jnx_pack_gate_up", "jnx_op_pack",
           "jnx_op_rmsnorm", "jnx_op_gemm_workspace_bytes", "jnx_op_gemm", "jnx_op_attention",
           "jnx_op_final_pool", "jnx_trace_enable", "jnx_trace_disable", "jnx_trace_count",
           "jnx_trace_read", "jnx_op_gemm_rope_noalloc", "jnx_op_gemm_rope_noalloc_status",
           "jnx_sched_poll", "jnx_diag_ex2_poly", "jnx_diag_bounded_wait",
           "jnx_heads_backward_accumulate", "jnx_heads_adamw", "jnx_heads_backward_adamw",
           "jnx_backbone_saved_bytes",
           "jnx_backbone_forward_train", "jnx_heads_backward_input", "jnx_transpose",
           "jnx_backbone_backward_workspace_bytes", "jnx_backbone_backward_lora",
           "jnx_op_attention_lse", "jnx_op_attention_backward_prep",
           "jnx_op_attention_backward_workspace_bytes", "jnx_op_attention_backward",
           "jnx_op_rms_backward", "jnx_op_gemm_glu_backward", "jnx_op_ffn_glu_backward", "jnx_flow_workspace_bytes",
           "jnx_flow_forward", "jnx_flow_backward", "jnx_flow_sample", "jnx_adamw_tensors")


def lib() -> C.CDLL:
    """Load libjnx.so (raises if it has not been built)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -m paper_2607_16074_gb300.build`")
    L = C.CDLL(LIB_PATH)
    vp, i32, i64, sz, f32 = C.c_void_p, C.c_int32, C.c_int64, C.c_size_t, C.c_float
    sig = {
        "jnx_last_error": (C.c_char_p, []),
        "jnx_version": (i32, []),
        "jnx_group_plan": (i32, [C.POINTER(jnx_schema), i32, C.POINTER(jnx_request), i32, i32,
                                 C.POINTER(jnx_limits), C.POINTER(jnx_plan)]),
        "jnx_group_attn_items": (i32, [C.POINTER(jnx_group), vp, i32]),
        "jnx_sched_poll": (i32, [C.POINTER(jnx_schema), i32, C.POINTER(jnx_request),
                                 C.POINTER(C.c_double), i32, i32, C.c_double,
                                 C.POINTER(jnx_sched_policy), P32, C.POINTER(C.c_int32),
                                 C.POINTER(C.c_double)]),
        "jnx_backbone_workspace_bytes": (sz, [C.POINTER(jnx_backbone), i32]),
        "jnx_backbone_forward": (i32, [C.POINTER(jnx_backbone), C.POINTER(jnx_group), vp, i64,
                                       vp, i64, vp, vp, vp, sz, vp]),
        "jnx_heads_workspace_bytes": (sz, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group)]),
        "jnx_heads_forward": (i32, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group), vp, vp, vp,
                                    vp, vp, vp, sz, vp]),
        "jnx_heads_backward": (i32, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group), vp, vp, vp,
                                     C.POINTER(jnx_head_grads), vp, sz, vp]),
        "jnx_heads_backward_accumulate": (i32, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group),
                                                vp, vp, vp, C.POINTER(jnx_head_grads), vp, sz,
                                                vp]),
        "jnx_heads_adamw": (i32, [C.POINTER(jnx_head), C.POINTER(jnx_head_grads),
                                  C.POINTER(jnx_head_opt), i32, C.POINTER(jnx_group),
                                  C.POINTER(jnx_adamw), vp]),
        "jnx_heads_backward_adamw": (i32, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group), vp, vp,
                                           vp, C.POINTER(jnx_head_grads), i32,
                                           C.POINTER(jnx_head_opt), C.POINTER(jnx_adamw), vp, vp,
                                           sz, vp]),
        "jnx_backbone_saved_bytes": (sz, [C.POINTER(jnx_backbone), i32]),
        "jnx_backbone_forward_train": (i32, [C.POINTER(jnx_backbone), C.POINTER(jnx_group), vp,
                                             i64, vp, i64, vp, vp, vp, vp, sz, vp]),
        "jnx_heads_backward_input": (i32, [C.POINTER(jnx_head), i32, C.POINTER(jnx_group), vp,
                                           vp, vp, C.POINTER(jnx_head_grads), vp, vp, sz, vp]),
        "jnx_transpose": (i32, [vp, i32, i32, i32, vp, vp]),
        "jnx_backbone_backward_workspace_bytes": (sz, [C.POINTER(jnx_backbone), i32]),
        "jnx_backbone_backward_lora": (i32, [C.POINTER(jnx_backbone), C.POINTER(jnx_layer_t),
                                             C.POINTER(jnx_group), vp, vp,
                                             C.POINTER(jnx_lora_grads), i32, vp, sz, vp]),
        "jnx_op_attention_lse": (i32, [vp, i32, i32, i32, i32, vp, i32, i32, vp, vp, vp, vp]),
        "jnx_op_attention_backward_prep": (i32, [vp, vp, i32, i32, i32, vp, vp, vp]),
        "jnx_op_attention_backward_workspace_bytes": (sz, [i32, i32, i32]),
        "jnx_op_attention_backward": (i32, [vp, vp, vp, vp, i32, i32, i32, i32, vp, vp, i32, i32,
                                            vp, f32, vp, vp, sz, vp, vp]),
        "jnx_op_rms_backward": (i32, [vp, vp, f32, vp, vp, i32, i32, vp, vp, vp]),
        "jnx_op_gemm_glu_backward": (i32, [vp, vp, i32, i32, i32, vp, i32, vp]),
        "jnx_op_ffn_glu_backward": (i32, [vp, vp, vp, vp, i32, i32, i32, i32, vp, vp]),
        "jnx_flow_workspace_bytes": (sz, [C.POINTER(jnx_flow_head), C.POINTER(jnx_group)]),
        "jnx_flow_forward": (i32, [C.POINTER(jnx_flow_head), C.POINTER(jnx_group), vp, vp, vp,
                                   vp, vp, vp, vp, sz, vp]),
        "jnx_flow_backward": (i32, [C.POINTER(jnx_flow_head), C.POINTER(jnx_group), vp,
                                    C.POINTER(jnx_flow_grads), i32, vp, sz, vp]),
        "jnx_flow_sample": (i32, [C.POINTER(jnx_flow_head), C.POINTER(jnx_group), vp, vp, i32,
                                  vp, vp, sz, vp]),
        "jnx_adamw_tensors": (i32, [C.POINTER(jnx_adam_tensor), i32, C.POINTER(jnx_adamw), vp]),
        "jnx_check_status": (i32, [vp, vp]),
        "jnx_pack_gate_up": (i32, [vp, vp, i32, i32, vp, vp]),
        "jnx_op_pack": (i32, [C.POINTER(jnx_group), vp, i64, vp, i64, vp, i32, i32, vp, vp, vp]),
        "jnx_op_rmsnorm": (i32, [vp, vp, f32, i32, i32, vp, vp]),
        "jnx_op_gemm_workspace_bytes": (sz, [i32, i32]),
        "jnx_op_gemm": (i32, [vp, vp, i32, i32, i32, i32, vp, i32, vp, i32, i32, i32, f32, i32,
                              vp, sz, vp]),
        "jnx_op_attention": (i32, [vp, i32, i32, i32, i32, vp, i32, i32, vp, vp, vp]),
        "jnx_op_final_pool": (i32, [vp, vp, f32, vp, i32, i32, vp, vp, vp]),
        "jnx_trace_enable": (i32, [i32]),
        "jnx_trace_disable": (i32, []),
        "jnx_trace_count": (i32, []),
        "jnx_trace_read": (i32, [vp, vp, vp, i32, P32]),
        "jnx_op_gemm_rope_noalloc": (i32, [vp, vp, i32, i32, i32, vp, i32, vp, i32, i32, i32, f32,
                                           vp]),
        "jnx_op_gemm_rope_noalloc_status": (i32, [vp]),
        "jnx_diag_ex2_poly": (i32, [vp, vp, i32, vp]),
        "jnx_diag_bounded_wait": (i32, [C.c_int64, i32, vp, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _LIB = L
    return L


def check(code: int) -> None:
    if code != JNX_OK:
        raise JnxError(code, lib().jnx_last_error().decode())


def jnx_last_error() -> str:
    return lib().jnx_last_error().decode()


def jnx_version() -> int:
    return lib().jnx_version()


# ---------------------------------------------------------------------------
# plan
# ---------------------------------------------------------------------------

class Plan:
    """Host result of jnx_group_plan: numpy int32 arrays trimmed to size."""

    FIELDS = ("cu_seqlens", "sample_slot", "sample_req", "sample_target", "sample_width",
              "seg_offsets", "slot_tenant", "gather_src", "pos_ids")

    def __init__(self, raw: jnx_plan, arrays: dict):
        self.n_requests = raw.n_requests
        self.n_samples = raw.n_samples
        self.n_tokens = raw.n_tokens
        self.n_slots = raw.n_slots
        self.max_seqlen = raw.max_seqlen
        S, N, G = raw.n_samples, raw.n_tokens, raw.n_slots
        size = dict(cu_seqlens=S + 1, sample_slot=S, sample_req=S, sample_target=S,
                    sample_width=S, seg_offsets=G + 1, slot_tenant=G, gather_src=N, pos_ids=N)
        for k in self.FIELDS:
            setattr(self, k, arrays[k][:size[k]].copy())

    def as_dict(self) -> dict:
        d = {k: getattr(self, k).tolist() for k in self.FIELDS}
        d.update(n_requests=self.n_requests, n_samples=self.n_samples, n_tokens=self.n_tokens,
                 n_slots=self.n_slots, max_seqlen=self.max_seqlen)
        return d


def make_schemas(schemas: Sequence[dict]):
    arr = (jnx_schema * max(1, len(schemas)))()
    for i, s in enumerate(schemas):
        arr[i] = jnx_schema(s["backbone_id"], s["d_model"], s["vision_tokens"], s["embed_dtype"],
                            s["vocab_id"], s["rope_id"], s["max_images"], s["action_width"])
    return arr


def make_requests(requests: Sequence[dict]):
    """requests: dicts with tenant, schema, samples (dicts n_img, text_len,
    vision_row, text_pos, target_off).  Returns (array, keepalive)."""
    keep = []
    arr = (jnx_request * max(1, len(requests)))()
    for i, r in enumerate(requests):
        ss = (jnx_sample * max(1, len(r["samples"])))()
        for j, s in enumerate(r["samples"]):
            ss[j] = jnx_sample(s["n_img"], s["text_len"], s.get("vision_row", 0),
                               s.get("text_pos", 0), s.get("target_off", 0))
        keep.append(ss)
        arr[i] = jnx_request(r["tenant"], r["schema"], len(r["samples"]), 0,
                             C.cast(ss, C.POINTER(jnx_sample)))
    return arr, keep


def jnx_group_plan(schemas: Sequence[dict], requests: Sequence[dict], n_tenants: int,
                   max_samples: int, max_tokens: int, caps=None) -> Plan:
    """Run the host plan; grows the output arrays once if they are too small."""
    L = lib()
    sch = make_schemas(schemas)
    req, keep = make_requests(requests)
    lim = jnx_limits(min(max_samples, 2**31 - 1), min(max_tokens, 2**31 - 1))
    cs, ct, cg = caps or (64, 4096, 8)
    for attempt in range(2):
        arrays = dict(cu_seqlens=np.zeros(cs + 1, np.int32), sample_slot=np.zeros(cs, np.int32),
                      sample_req=np.zeros(cs, np.int32), sample_target=np.zeros(cs, np.int32),
                      sample_width=np.zeros(cs, np.int32), seg_offsets=np.zeros(cg + 1, np.int32),
                      slot_tenant=np.zeros(cg, np.int32), gather_src=np.zeros(max(ct, 1), np.int32),
                      pos_ids=np.zeros(max(ct, 1), np.int32))
        raw = jnx_plan(cs, ct, cg, 0, 0, 0, 0, 0,
                       *[arrays[k].ctypes.data_as(P32) for k in Plan.FIELDS])
        rc = L.jnx_group_plan(sch, len(schemas), req, len(requests), n_tenants, C.byref(lim),
                              C.byref(raw))
        if rc == JNX_ERR_CAPACITY and attempt == 0:
            cs, ct, cg = max(raw.n_samples, 1), max(raw.n_tokens, 1), max(raw.n_slots, 1)
            continue
        check(rc)
        return Plan(raw, arrays)
    raise JnxError(JNX_ERR_CAPACITY, "plan capacity")


def jnx_sched_poll(schemas: Sequence[dict], requests: Sequence[dict], arrival: Sequence[float],
                   n_tenants: int, now: float, timeout: float, batch_samples: int,
                   max_tokens: int, skip_ahead: bool = False):
    """The inference scheduler's decision at `now`: (take, wake) with take
    the ascending queue indices to run now (empty: not yet) and wake the
    time to poll again when not firing (`now` when firing, inf when empty)."""
    L = lib()
    sch = make_schemas(schemas)
    req, keep = make_requests(requests)
    n = len(requests)
    arr = (C.c_double * max(1, n))(*[float(a) for a in arrival])
    take = np.zeros(max(1, n), np.int32)
    n_take, wake = C.c_int32(0), C.c_double(0.0)
    pol = jnx_sched_policy(float(timeout), min(int(batch_samples), 2**31 - 1),
                           min(int(max_tokens), 2**31 - 1), int(bool(skip_ahead)), 0)
    check(L.jnx_sched_poll(sch, len(schemas), req, arr, n, n_tenants, float(now), C.byref(pol),
                           take.ctypes.data_as(P32), C.byref(n_take), C.byref(wake)))
    return take[:n_take.value].tolist(), wake.value


# ---------------------------------------------------------------------------
# tracing
# ---------------------------------------------------------------------------
KERNEL_NAMES = {1: "pack", 2: "rmsnorm", 3: "gemm_qkv_rope", 4: "attention", 5: "gemm_o_resid",
                6: "gemm_gate_up_glu", 7: "gemm_down_resid", 8: "final_norm_pool",
                9: "rope_table", 10: "heads_fwd", 11: "heads_bwd", 12: "gemm", 13: "lora_down",
                14: "heads_adamw", 15: "gemm_bwd", 16: "attention_bwd", 17: "norm_bwd",
                18: "lora_bwd", 19: "flow_gemm", 20: "flow_attention", 21: "flow_misc",
                22: "flow_wgrad"}
TENSOR_KERNELS = (3, 4, 5, 6, 7, 12, 13, 15, 16, 18, 19, 20, 22)


def jnx_trace_enable(capacity: int) -> None:
    check(lib().jnx_trace_enable(capacity))


def jnx_trace_disable() -> None:
    check(lib().jnx_trace_disable())


def jnx_trace_count() -> int:
    return lib().jnx_trace_count()


def jnx_trace_read(cap: int):
    """(kinds, ms, work) numpy arrays of the recorded launches."""
    kinds = np.zeros(cap, np.int32)
    ms = np.zeros(cap, np.float32)
    work = np.zeros(cap, np.float64)
    n = C.c_int32(0)
    check(lib().jnx_trace_read(kinds.ctypes.data, ms.ctypes.data, work.ctypes.data, cap,
                               C.byref(n)))
    return kinds[:n.value], ms[:n.value], work[:n.value]
