"""Device-side plumbing around the C ABI: PyTorch holds the device memory and
the stream; these classes only fill the C structs with its addresses and
call the library.  No arithmetic of the method happens here.
"""
from __future__ import annotations

import ctypes as C
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

from . import jnx as J


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream(stream: Optional[torch.cuda.Stream]) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


class DeviceGroup:
    """A plan's arrays copied to the device, wrapped in a jnx_group."""

    DEV = ("cu_seqlens", "sample_slot", "sample_target", "seg_offsets", "gather_src", "pos_ids")

    def __init__(self, plan: J.Plan, device="cuda", non_blocking: bool = False):
        self.plan = plan
        self.h = {k: np.ascontiguousarray(getattr(plan, k), dtype=np.int32)
                  for k in ("cu_seqlens", "seg_offsets", "slot_tenant")}
        self.d = {}
        for k in self.DEV:
            a = torch.from_numpy(np.ascontiguousarray(getattr(plan, k), dtype=np.int32))
            if non_blocking:
                a = a.pin_memory()
            self.d[k] = a.to(device, non_blocking=non_blocking)
        hp = lambda k: self.h[k].ctypes.data_as(J.P32)
        self.struct = J.jnx_group(
            plan.n_samples, plan.n_tokens, plan.n_slots, plan.max_seqlen,
            *[self.d[k].data_ptr() or None for k in self.DEV],
            hp("cu_seqlens"), hp("seg_offsets"), hp("slot_tenant"), None, 0)
        # the attention work list on the device too, so the backbone's calls
        # read it instead of uploading it (and can be captured into a graph)
        L = J.lib()
        n = L.jnx_group_attn_items(C.byref(self.struct), None, 0)
        if n < 0:
            J.check(n)
        items = np.zeros(2 * max(n, 1), dtype=np.int32)
        got = L.jnx_group_attn_items(C.byref(self.struct), items.ctypes.data, n)
        if got != n:
            J.check(got if got < 0 else J.JNX_ERR_INVALID_ARG)
        t = torch.from_numpy(items)
        if non_blocking:
            t = t.pin_memory()
        self.d["attn_items"] = t.to(device, non_blocking=non_blocking)
        self.struct.attn_items = self.d["attn_items"].data_ptr() if n else None
        self.struct.n_attn_items = n

    @property
    def ref(self):
        return C.byref(self.struct)


class DeviceBackbone:
    """Frozen backbone weights on the device in the library's layout: the
    fused [W_q; W_k; W_v] rows and the 128-row interleaved gate/up matrix
    (built by jnx_pack_gate_up)."""

    def __init__(self, cfg, weights: Dict, n_tenants: int = 1, stream=None):
        self.cfg = cfg
        L = J.lib()
        self.keep: List[torch.Tensor] = []
        self.layers = (J.jnx_layer * max(1, cfg.n_layers))()
        s = _stream(stream)
        for i, lw in enumerate(weights["layers"]):
            w_qkv = torch.cat([lw["wq"], lw["wk"], lw["wv"]], dim=0).contiguous()
            w_gu = torch.empty((2 * cfg.d_ff, cfg.d), dtype=torch.bfloat16, device=w_qkv.device)
            J.check(L.jnx_pack_gate_up(lw["wg"].data_ptr(), lw["wu"].data_ptr(), cfg.d_ff, cfg.d,
                                       w_gu.data_ptr(), s))
            ent = dict(attn_norm=lw["attn_norm"], w_qkv=w_qkv, w_o=lw["wo"],
                       ffn_norm=lw["ffn_norm"], w_gu=w_gu, w_down=lw["wd"])
            names = ["attn_norm", "w_qkv", "w_o", "ffn_norm", "w_gu", "w_down"]
            if cfg.lora_rank:
                for p in ("q", "k", "v", "o"):
                    ent["lora_a_" + p] = lw["lora_a_" + p].contiguous()
                    ent["lora_b_" + p] = lw["lora_b_" + p].contiguous()
                    names += ["lora_a_" + p, "lora_b_" + p]
            self.keep += list(ent.values())
            self.layers[i] = J.jnx_layer(**{k: ent[k].data_ptr() for k in names})
        self.text_table = weights["text_table"]
        self.final_norm = weights["final_norm"]
        self.struct = J.jnx_backbone(cfg.n_layers, cfg.d, cfg.n_heads, cfg.n_kv_heads,
                                     cfg.head_dim, cfg.d_ff, cfg.glu, cfg.lora_rank, n_tenants,
                                     cfg.vocab, cfg.vision_tokens, cfg.eps, cfg.rope_theta,
                                     self.text_table.data_ptr(), self.final_norm.data_ptr(),
                                     C.cast(self.layers, C.POINTER(J.jnx_layer)))

    def workspace_bytes(self, n_tokens: int) -> int:
        return J.lib().jnx_backbone_workspace_bytes(C.byref(self.struct), n_tokens)

    def forward(self, group: DeviceGroup, vision: torch.Tensor, text_ids: torch.Tensor,
                pooled: Optional[torch.Tensor], hidden: Optional[torch.Tensor],
                ws: torch.Tensor, stream=None) -> None:
        J.check(J.lib().jnx_backbone_forward(
            C.byref(self.struct), group.ref, vision.data_ptr(), vision.shape[0],
            text_ids.data_ptr(), text_ids.shape[0], _ptr(pooled), _ptr(hidden),
            ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)))

    # ---- trainable adapters ------------------------------------------------
    def saved_bytes(self, n_tokens: int) -> int:
        return J.lib().jnx_backbone_saved_bytes(C.byref(self.struct), n_tokens)

    def backward_workspace_bytes(self, n_tokens: int) -> int:
        return J.lib().jnx_backbone_backward_workspace_bytes(C.byref(self.struct), n_tokens)

    def prepare_backward(self, stream=None) -> None:
        """Transposed copies of the frozen weights (built once on the device)
        and zeroed fp32 adapter-gradient buffers, one set per layer."""
        cfg, L, s = self.cfg, J.lib(), _stream(stream)
        n = max(1, cfg.n_layers)
        self.layers_t = (J.jnx_layer_t * n)()
        self.lgarr = (J.jnx_lora_grads * n)()
        self.keep_t: List[torch.Tensor] = []
        self.lora_grads: List[Dict[str, torch.Tensor]] = []
        per = len(self.keep) // max(1, cfg.n_layers)
        for i in range(cfg.n_layers):
            ent = self.keep[i * per:(i + 1) * per]
            w_qkv, w_o, w_gu, w_down = ent[1], ent[2], ent[4], ent[5]
            outs = []
            for w in (w_qkv, w_o, w_gu, w_down):
                t = torch.empty((w.shape[1], w.shape[0]), dtype=torch.bfloat16, device=w.device)
                J.check(L.jnx_transpose(w.data_ptr(), 1, w.shape[0], w.shape[1], t.data_ptr(), s))
                outs.append(t)
            self.keep_t += outs
            self.layers_t[i] = J.jnx_layer_t(*[t.data_ptr() for t in outs])
            lw = dict(zip(["attn_norm", "w_qkv", "w_o", "ffn_norm", "w_gu", "w_down",
                           "lora_a_q", "lora_b_q", "lora_a_k", "lora_b_k", "lora_a_v",
                           "lora_b_v", "lora_a_o", "lora_b_o"], ent))
            g = {}
            for name in J.LORA_GRADS:
                src = lw.get("lora_" + name)
                g[name] = (torch.zeros(src.shape, dtype=torch.float32, device=src.device)
                           if src is not None else None)
            self.lora_grads.append(g)
            self.lgarr[i] = J.jnx_lora_grads(*[_ptr(g[k]) for k in J.LORA_GRADS])

    def lora_pairs(self):
        """(adapter [n_tenants, ...] bf16, its gradient buffer) of every layer,
        for TenantAdamW (the adapters are updated in place)."""
        per = len(self.keep) // max(1, self.cfg.n_layers)
        out = []
        for i in range(self.cfg.n_layers):
            ent = self.keep[i * per:(i + 1) * per][6:]
            for name, p in zip(J.LORA_GRADS, ent):
                out.append((p, self.lora_grads[i][name]))
        return out

    def forward_train(self, group: DeviceGroup, vision, text_ids, pooled, hidden, saved, ws,
                      stream=None) -> None:
        J.check(J.lib().jnx_backbone_forward_train(
            C.byref(self.struct), group.ref, vision.data_ptr(), vision.shape[0],
            text_ids.data_ptr(), text_ids.shape[0], _ptr(pooled), _ptr(hidden),
            saved.data_ptr(), ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)))

    def backward_lora(self, group: DeviceGroup, saved, d_hidden, ws, accumulate: bool = False,
                      stream=None) -> None:
        """Every group tenant's adapter gradients into self.lora_grads (its
        slice only), from dloss/d(final normed rows)."""
        J.check(J.lib().jnx_backbone_backward_lora(
            C.byref(self.struct), self.layers_t, group.ref, saved.data_ptr(), d_hidden.data_ptr(),
            self.lgarr, 1 if accumulate else 0, ws.data_ptr(), ws.numel() * ws.element_size(),
            _stream(stream)))


class DeviceHeads:
    """One head slot per tenant (bf16 parameters) and fp32 gradient slots."""

    def __init__(self, tenants: Sequence, d: int, heads: List[Dict], device="cuda"):
        n = len(tenants)
        self.n = n
        self.arr = (J.jnx_head * max(1, n))()
        self.garr = (J.jnx_head_grads * max(1, n))()
        self.grads: List[Dict[str, torch.Tensor]] = []
        self.keep = []
        for t, (tn, hw) in enumerate(zip(tenants, heads)):
            if tn.head_kind == J.JNX_HEAD_MLP:
                self.arr[t] = J.jnx_head(tn.head_kind, d, tn.d_hidden, 0, 0, tn.width,
                                         hw["w1"].data_ptr(), hw["b1"].data_ptr(),
                                         hw["w2"].data_ptr(), hw["b2"].data_ptr(),
                                         None, None, None, None, None)
                g = {k: torch.zeros(hw[k].shape, dtype=torch.float32, device=device)
                     for k in ("w1", "b1", "w2", "b2")}
                self.garr[t] = J.jnx_head_grads(*[g[k].data_ptr() for k in ("w1", "b1", "w2",
                                                                             "b2")],
                                                None, None, None, None, None)
            else:
                self.arr[t] = J.jnx_head(tn.head_kind, d, 0, tn.n_queries, tn.q_dim, tn.width,
                                         None, None, None, None, hw["q"].data_ptr(),
                                         hw["wk"].data_ptr(), hw["wv"].data_ptr(),
                                         hw["wout"].data_ptr(), hw["bout"].data_ptr())
                g = {k: torch.zeros(hw[k].shape, dtype=torch.float32, device=device)
                     for k in ("q", "wk", "wv", "wout", "bout")}
                self.garr[t] = J.jnx_head_grads(None, None, None, None,
                                                *[g[k].data_ptr() for k in ("q", "wk", "wv",
                                                                            "wout", "bout")])
            self.grads.append(g)
            self.keep.append(hw)

    def workspace_bytes(self, group: DeviceGroup) -> int:
        return J.lib().jnx_heads_workspace_bytes(self.arr, self.n, group.ref)

    def forward(self, group: DeviceGroup, pooled, hidden, targets, preds, loss, ws,
                stream=None) -> None:
        """targets and loss may both be None (inference: predictions only)."""
        J.check(J.lib().jnx_heads_forward(
            self.arr, self.n, group.ref, _ptr(pooled), _ptr(hidden), _ptr(targets),
            preds.data_ptr(), _ptr(loss), ws.data_ptr(), ws.numel() * ws.element_size(),
            _stream(stream)))

    def backward(self, group: DeviceGroup, pooled, hidden, targets, ws, stream=None,
                 accumulate: bool = False) -> None:
        """Gradients into each group tenant's slot: overwritten, or added to
        what is there (gradient accumulation) with accumulate=True."""
        fn = J.lib().jnx_heads_backward_accumulate if accumulate else J.lib().jnx_heads_backward
        J.check(fn(self.arr, self.n, group.ref, _ptr(pooled), _ptr(hidden), targets.data_ptr(),
                   self.garr, ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)))

    def backward_input(self, group: DeviceGroup, pooled, hidden, targets, d_hidden, ws,
                       stream=None) -> None:
        """backward, and also dloss/d(final normed row) of every token row."""
        J.check(J.lib().jnx_heads_backward_input(
            self.arr, self.n, group.ref, _ptr(pooled), _ptr(hidden), targets.data_ptr(),
            self.garr, d_hidden.data_ptr(), ws.data_ptr(), ws.numel() * ws.element_size(),
            _stream(stream)))

    def init_optimizer(self) -> None:
        """Tenant-private AdamW state: an fp32 master copy of every head
        parameter (from its bf16 value) and zero moments, per tenant."""
        self.opt = (J.jnx_head_opt * max(1, self.n))()
        self.opt_state: List[Dict[str, Dict[str, torch.Tensor]]] = []
        for t, hw in enumerate(self.keep):
            st = {}
            for k, name in enumerate(J.HEAD_PARAMS):
                if name not in hw:
                    continue
                p = hw[name]
                st[name] = dict(master=p.float().clone(), m=torch.zeros_like(p, dtype=torch.float32),
                                v=torch.zeros_like(p, dtype=torch.float32))
                self.opt[t].master[k] = st[name]["master"].data_ptr()
                self.opt[t].m[k] = st[name]["m"].data_ptr()
                self.opt[t].v[k] = st[name]["v"].data_ptr()
            self.opt_state.append(st)

    def adamw_step(self, group: DeviceGroup, lr: float, beta1: float = 0.9,
                   beta2: float = 0.999, eps: float = 1e-8, weight_decay: float = 0.0,
                   stream=None) -> None:
        """One AdamW step on every group tenant's head from its gradients
        (bf16 parameters updated in place; the tenant's step and policy
        version counters increment)."""
        hp = J.jnx_adamw(lr, beta1, beta2, eps, weight_decay)
        J.check(J.lib().jnx_heads_adamw(self.arr, self.garr, self.opt, self.n, group.ref,
                                        C.byref(hp), _stream(stream)))

    def backward_adamw(self, group: DeviceGroup, pooled, hidden, targets, ws, lr: float,
                       beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8,
                       weight_decay: float = 0.0, accumulate: bool = False, d_hidden=None,
                       stream=None) -> None:
        """The heads backward with every group tenant's AdamW step fused into
        it: the same result as backward() then adamw_step(), without storing
        the gradients (with accumulate=True the gradients already in the
        slots are added first).  d_hidden, if given, receives the gradient at
        the final normed rows (as backward_input)."""
        hp = J.jnx_adamw(lr, beta1, beta2, eps, weight_decay)
        J.check(J.lib().jnx_heads_backward_adamw(
            self.arr, self.n, group.ref, _ptr(pooled), _ptr(hidden), _ptr(targets), self.garr,
            1 if accumulate else 0, self.opt, C.byref(hp), _ptr(d_hidden), ws.data_ptr(),
            ws.numel() * ws.element_size(), _stream(stream)))

    def version(self, t: int) -> int:
        return int(self.opt[t].version)


class DeviceFlowHeads:
    """Flow-matching action experts (DiT heads) of n_tenants tenants with the
    same dimensions: stacked bf16 parameters (the gate/up pair of each block
    packed by jnx_pack_gate_up) and fp32 gradient buffers of the same shapes."""

    def __init__(self, dims: Dict, weights: Dict, stream=None):
        L, s = J.lib(), _stream(stream)
        self.dims = dims
        T, dm, F = dims["n_tenants"], dims["d_model"], dims["d_ff"]
        self.keep = {k: weights[k].contiguous() for k in J.FLOW_PARAMS}
        self.blocks = []
        for B in weights["blocks"]:
            w_gu = torch.empty((T, 2 * F, dm), dtype=torch.bfloat16, device=B["wg"].device)
            for t in range(T):
                J.check(L.jnx_pack_gate_up(B["wg"][t].contiguous().data_ptr(),
                                           B["wu"][t].contiguous().data_ptr(), F, dm,
                                           w_gu[t].data_ptr(), s))
            self.blocks.append(dict(w_qkv=B["w_qkv"].contiguous(), w_kvc=B["w_kvc"].contiguous(),
                                    w_o=B["w_o"].contiguous(), w_gu=w_gu,
                                    w_d=B["w_d"].contiguous()))
        nb = max(1, len(self.blocks))
        self.barr = (J.jnx_flow_block * nb)(*[J.jnx_flow_block(
            *[b[k].data_ptr() for k in J.FLOW_BLOCK_PARAMS]) for b in self.blocks])
        self.struct = J.jnx_flow_head(
            dm, F, len(self.blocks), dims["chunk"], dims["action_dim"], dims["d_in"], T,
            *[self.keep[k].data_ptr() for k in J.FLOW_PARAMS],
            C.cast(self.barr, C.POINTER(J.jnx_flow_block)))
        dev = self.keep["w_in"].device
        self.grads = {k: torch.zeros(self.keep[k].shape, dtype=torch.float32, device=dev)
                      for k in J.FLOW_PARAMS}
        self.block_grads = [{k: torch.zeros(b[k].shape, dtype=torch.float32, device=dev)
                             for k in J.FLOW_BLOCK_PARAMS} for b in self.blocks]
        self.bgarr = (J.jnx_flow_block_grads * nb)(*[J.jnx_flow_block_grads(
            *[g[k].data_ptr() for k in J.FLOW_BLOCK_PARAMS]) for g in self.block_grads])
        self.gstruct = J.jnx_flow_grads(*[self.grads[k].data_ptr() for k in J.FLOW_PARAMS],
                                        C.cast(self.bgarr, C.POINTER(J.jnx_flow_block_grads)))

    def workspace_bytes(self, group: DeviceGroup) -> int:
        return J.lib().jnx_flow_workspace_bytes(C.byref(self.struct), group.ref)

    def param_pairs(self):
        """(stacked parameter, its gradient buffer) of every expert tensor
        (the packed gate/up pair as one), for TenantAdamW."""
        out = [(self.keep[k], self.grads[k]) for k in J.FLOW_PARAMS]
        for b, g in zip(self.blocks, self.block_grads):
            out += [(b[k], g[k]) for k in J.FLOW_BLOCK_PARAMS]
        return out

    def forward(self, group: DeviceGroup, hidden, actions, noise, tau, velocity, loss, ws,
                stream=None) -> None:
        J.check(J.lib().jnx_flow_forward(
            C.byref(self.struct), group.ref, hidden.data_ptr(), actions.data_ptr(),
            noise.data_ptr(), tau.data_ptr(), velocity.data_ptr(), loss.data_ptr(),
            ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)))

    def backward(self, group: DeviceGroup, hidden, ws, accumulate: bool = False,
                 stream=None) -> None:
        J.check(J.lib().jnx_flow_backward(
            C.byref(self.struct), group.ref, hidden.data_ptr(), C.byref(self.gstruct),
            1 if accumulate else 0, ws.data_ptr(), ws.numel() * ws.element_size(),
            _stream(stream)))

    def sample(self, group: DeviceGroup, hidden, noise, n_steps: int, actions, ws,
               stream=None) -> None:
        J.check(J.lib().jnx_flow_sample(
            C.byref(self.struct), group.ref, hidden.data_ptr(), noise.data_ptr(), n_steps,
            actions.data_ptr(), ws.data_ptr(), ws.numel() * ws.element_size(), _stream(stream)))


class TenantAdamW:
    """Tenant-private AdamW over stacked per-tenant parameters: for every
    (parameter [n_tenants, ...] bf16, gradient [n_tenants, ...] fp32) pair an
    fp32 master copy and zero moments; step(tenants) updates only those
    tenants' slices, each slice with its own step counter
    (jnx_adamw_tensors)."""

    def __init__(self, pairs):
        self.pairs = [(p, g) for p, g in pairs]
        self.master = [p.float().clone() for p, _ in self.pairs]
        self.m = [torch.zeros_like(x) for x in self.master]
        self.v = [torch.zeros_like(x) for x in self.master]
        self.counts: Dict = {}

    def steps(self, i: int, t: int) -> int:
        c = self.counts.get((i, t))
        return int(c.value) if c is not None else 0

    def step(self, tenants, lr: float, beta1: float = 0.9, beta2: float = 0.999,
             eps: float = 1e-8, weight_decay: float = 0.0, stream=None) -> None:
        arr = []
        for i, (p, g) in enumerate(self.pairs):
            for t in tenants:
                cnt = self.counts.setdefault((i, t), C.c_int32(0))
                arr.append(J.jnx_adam_tensor(p[t].data_ptr(), self.master[i][t].data_ptr(),
                                             self.m[i][t].data_ptr(), self.v[i][t].data_ptr(),
                                             g[t].data_ptr(), p[t].numel(), C.pointer(cnt)))
        tab = (J.jnx_adam_tensor * max(1, len(arr)))(*arr)
        hp = J.jnx_adamw(lr, beta1, beta2, eps, weight_decay)
        J.check(J.lib().jnx_adamw_tensors(tab, len(arr), C.byref(hp), _stream(stream)))


def check_status(ws: torch.Tensor, stream=None) -> None:
    J.check(J.lib().jnx_check_status(ws.data_ptr(), _stream(stream)))


class GroupedStep:
    """One grouped step through the C ABI: backbone forward over the packed
    batch, then every group tenant's head forward, loss and backward."""

    def __init__(self, backbone: DeviceBackbone, heads: DeviceHeads, group: DeviceGroup,
                 device="cuda"):
        self.bb, self.heads, self.group = backbone, heads, group
        cfg = backbone.cfg
        S, N = group.plan.n_samples, group.plan.n_tokens
        kinds = {heads.arr[t].kind for t in group.plan.slot_tenant.tolist()}
        self.need_hidden = J.JNX_HEAD_XATTN in kinds
        self.need_pooled = J.JNX_HEAD_MLP in kinds or not kinds
        self.pooled = torch.zeros((max(S, 1), cfg.d), dtype=torch.float32, device=device)
        self.hidden = (torch.zeros((max(N, 1), cfg.d), dtype=torch.bfloat16, device=device)
                       if self.need_hidden else None)
        self.ws_bb = torch.zeros(max(backbone.workspace_bytes(N), 256), dtype=torch.uint8,
                                 device=device)
        self.ws_h = torch.zeros(max(heads.workspace_bytes(group), 256), dtype=torch.uint8,
                                device=device)
        self.loss = torch.full((max(heads.n, 1),), float("nan"), dtype=torch.float32, device=device)

    def run(self, vision, text_ids, targets, preds, stream=None) -> None:
        self.bb.forward(self.group, vision, text_ids,
                        self.pooled if self.need_pooled else None, self.hidden, self.ws_bb, stream)
        self.heads.forward(self.group, self.pooled, self.hidden, targets, preds, self.loss,
                           self.ws_h, stream)
        self.heads.backward(self.group, self.pooled, self.hidden, targets, self.ws_h, stream)

    def infer(self, vision, text_ids, preds, stream=None) -> None:
        """Inference: the shared backbone forward and every group tenant's
        head forward (predictions only; no targets, loss or backward)."""
        self.bb.forward(self.group, vision, text_ids,
                        self.pooled if self.need_pooled else None, self.hidden, self.ws_bb, stream)
        self.heads.forward(self.group, self.pooled, self.hidden, None, preds, None, self.ws_h,
                           stream)


class LoraTrainStep(GroupedStep):
    """One grouped training step of the tenants' adapters and heads through
    the C ABI: the shared forward keeping each block's residual input, every
    group tenant's head forward, loss and backward (with the gradient at its
    features), then the adapter backward through the frozen backbone.  Head
    gradients land in heads.grads, adapter gradients in backbone.lora_grads,
    each tenant's in its own slice."""

    def __init__(self, backbone: DeviceBackbone, heads: DeviceHeads, group: DeviceGroup,
                 device="cuda"):
        super().__init__(backbone, heads, group, device)
        if not hasattr(backbone, "layers_t"):
            backbone.prepare_backward()
        N, d = group.plan.n_tokens, backbone.cfg.d
        self.saved = torch.empty(max(backbone.saved_bytes(N) // 4, 1), dtype=torch.float32,
                                 device=device)
        self.d_hidden = torch.zeros((max(N, 1), d), dtype=torch.float32, device=device)
        self.ws_bwd = torch.zeros(max(backbone.backward_workspace_bytes(N), 256),
                                  dtype=torch.uint8, device=device)

    def run(self, vision, text_ids, targets, preds, stream=None, accumulate: bool = False) -> None:
        self.bb.forward_train(self.group, vision, text_ids,
                              self.pooled if self.need_pooled else None, self.hidden, self.saved,
                              self.ws_bb, stream)
        self.heads.forward(self.group, self.pooled, self.hidden, targets, preds, self.loss,
                           self.ws_h, stream)
        self.heads.backward_input(self.group, self.pooled, self.hidden, targets, self.d_hidden,
                                  self.ws_h, stream)
        self.bb.backward_lora(self.group, self.saved, self.d_hidden, self.ws_bwd,
                              accumulate=accumulate, stream=stream)


class StepPipeline:
    """Grouped steps fed from pinned host memory, each step's preparation
    overlapped with the step before it.

    While step i runs on the compute stream, the host plans step i+1 and a
    copy stream moves its inputs into the second of two device input
    buffers; step i+1 waits only for that copy (and its group's plan arrays,
    which go up on the compute stream behind step i).  Every step's per-slot
    loss and predictions come back to pinned host memory on the compute
    stream and are handed to `on_result(i, loss, preds)` once step i is done
    (while step i+1 is already queued on the GPU).  All steps share the
    GroupedStep's buffers and workspaces, so each step's group must need no
    more than the group the GroupedStep was built for."""

    def __init__(self, step: GroupedStep, vision_rows: int, n_text: int, targets_shape,
                 device="cuda"):
        self.step = step
        self.dev = device
        d = step.bb.cfg.d
        self.vis = [torch.empty((max(vision_rows, 1), d), dtype=torch.bfloat16, device=device)
                    for _ in range(2)]
        self.tid = [torch.empty(max(n_text, 1), dtype=torch.int32, device=device)
                    for _ in range(2)]
        self.tgt = [torch.empty(targets_shape, dtype=torch.float32, device=device)
                    for _ in range(2)]
        self.preds = torch.zeros(targets_shape, dtype=torch.float32, device=device)
        self.copy_stream = torch.cuda.Stream(device=device)
        self.copied = [torch.cuda.Event() for _ in range(2)]
        self.done = [torch.cuda.Event() for _ in range(2)]
        self.loss_h = [torch.empty(step.loss.shape, dtype=torch.float32).pin_memory()
                       for _ in range(2)]
        self.preds_h = [torch.empty(targets_shape, dtype=torch.float32).pin_memory()
                        for _ in range(2)]
        self.groups: List[Optional[DeviceGroup]] = [None, None]
        self.h2d_bytes = 0
        self.max_tokens = step.group.plan.n_tokens
        self.max_samples = step.group.plan.n_samples

    def _fits(self, g: DeviceGroup) -> None:
        s = self.step
        if (g.plan.n_tokens > self.max_tokens or g.plan.n_samples > self.max_samples
                or s.ws_h.numel() < s.heads.workspace_bytes(g)
                or s.ws_bb.numel() < s.bb.workspace_bytes(g.plan.n_tokens)):
            raise ValueError("StepPipeline: a step's group is larger than the step's buffers")
        kinds = {s.heads.arr[t].kind for t in g.plan.slot_tenant.tolist()}
        if ((J.JNX_HEAD_XATTN in kinds and not s.need_hidden)
                or (J.JNX_HEAD_MLP in kinds and not s.need_pooled)):
            raise ValueError("StepPipeline: a step's group has a head kind the step was not built for")

    def _stage(self, i: int, host: Dict[str, torch.Tensor], plan) -> None:
        b = i & 1
        g = DeviceGroup(plan, device=self.dev, non_blocking=True)
        self._fits(g)
        cs = self.copy_stream
        cs.wait_event(self.done[b])  # step i-2 has finished reading buffer b
        with torch.cuda.stream(cs):
            for dst, k in ((self.vis[b], "vision"), (self.tid[b], "text_ids"),
                           (self.tgt[b], "targets")):
                src = host[k]
                dst.view(-1)[:src.numel()].copy_(src.view(-1), non_blocking=True)
                self.h2d_bytes += src.numel() * src.element_size()
        self.copied[b].record(cs)
        self.groups[b] = g

    def run(self, batches: Sequence[Dict[str, torch.Tensor]], plan_fn, on_result=None) -> None:
        """batches[i]: pinned host tensors 'vision', 'text_ids', 'targets' of
        step i; plan_fn(i) returns step i's plan (called on the host while
        step i-1 runs)."""
        ks = torch.cuda.current_stream(self.dev)
        n = len(batches)
        if n == 0:
            return
        self._stage(0, batches[0], plan_fn(0))
        for i in range(n):
            b = i & 1
            ks.wait_event(self.copied[b])
            self.step.group = self.groups[b]
            self.step.run(self.vis[b], self.tid[b], self.tgt[b], self.preds, ks)
            self.loss_h[b].copy_(self.step.loss, non_blocking=True)
            self.preds_h[b].copy_(self.preds, non_blocking=True)
            self.done[b].record(ks)
            if i >= 1:
                self.done[b ^ 1].synchronize()
                if on_result is not None:
                    on_result(i - 1, self.loss_h[b ^ 1], self.preds_h[b ^ 1])
            if i + 1 < n:
                self._stage(i + 1, batches[i + 1], plan_fn(i + 1))
        self.done[(n - 1) & 1].synchronize()
        if on_result is not None:
            on_result(n - 1, self.loss_h[(n - 1) & 1], self.preds_h[(n - 1) & 1])
