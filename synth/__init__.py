"""Seeded synthetic workloads for the grouped multi-tenant path.

This module only draws random inputs and describes their shapes.  It holds
none of the method's arithmetic: no planning, no packing, no model math.  Both
the fp64 oracle (through the tests) and the CUDA path receive the arrays made
here, so the two sides always see identical inputs.

The five workloads follow the shapes of the group-batching experiment (§5.2)
and of the model families the paper runs there (a QwenOFT-like linear head, a
PaliGemma-2B-like MQA backbone with a query head, a 7B Llama-like backbone):

  tiny     2 tenants x 4 samples, 1 block, d=256 (64 vision rows + 16/24 text)
  small    8 tenants x U{8..32} samples, 6 blocks, d=1024
  mqa2b    16 tenants x 16 samples, 18 blocks, d=2048, 8x256 heads, 1 KV head,
           GeGLU 16384, 1-3 images per sample, cross-attention query heads
  zipf2b   64 tenants, Zipf(1.2) sample counts summing to 512, lengths
           260..840, LoRA rank 16 on Q/K/V/O, otherwise as mqa2b
  llama7b  32 tenants, ~64k packed tokens, 32 blocks, d=4096, 32x128 heads,
           SwiGLU 11008, MLP heads 4096->1024->56

Samples of a tenant arrive as requests of up to ``req_batch`` samples; the
requests of all tenants are interleaved round-robin in arrival (FIFO) order,
which is the order the Inference Queue sees them in (App. A, "Inference Queue
Composition").
"""
from __future__ import annotations

import dataclasses
import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional

import numpy as np

HEAD_MLP = 0
HEAD_XATTN = 1
GLU_SWIGLU = 0
GLU_GEGLU = 1


@dataclass
class Backbone:
    n_layers: int
    d: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    glu: int = GLU_SWIGLU
    lora_rank: int = 0
    eps: float = 1e-6
    rope_theta: float = 10000.0
    vocab: int = 32000
    vision_tokens: int = 256  # rows per image
    backbone_id: int = 0
    qk_std: float = 0.02     # std of W_q / W_k (a "sharp" test raises it)


@dataclass
class Tenant:
    head_kind: int
    chunk: int        # C, action chunk length
    action_dim: int   # D_t
    d_hidden: int = 0  # MLP hidden width
    n_queries: int = 32  # query head: learned action queries
    q_dim: int = 256      # query head: attention width
    max_images: int = 3

    @property
    def width(self) -> int:
        return self.chunk * self.action_dim


@dataclass
class Sample:
    n_img: int
    text_len: int
    vision_row: int = 0   # first row of this sample's vision embeddings
    text_pos: int = 0     # first position of its text ids
    target_off: int = 0   # first float of its action target / prediction

    def length(self, vision_tokens: int) -> int:
        return self.n_img * vision_tokens + self.text_len


@dataclass
class Request:
    tenant: int
    schema: int
    samples: List[Sample]


@dataclass
class Workload:
    name: str
    seed: int
    backbone: Backbone
    tenants: List[Tenant]
    requests: List[Request]
    max_samples: int = 1 << 30
    max_tokens: int = 1 << 30

    # ---- derived sizes -------------------------------------------------
    @property
    def samples(self) -> List[Sample]:
        return [s for r in self.requests for s in r.samples]

    @property
    def n_vision_rows(self) -> int:
        return sum(s.n_img for s in self.samples) * self.backbone.vision_tokens

    @property
    def n_text(self) -> int:
        return sum(s.text_len for s in self.samples)

    @property
    def n_target(self) -> int:
        return sum(self.tenants[r.tenant].width * len(r.samples) for r in self.requests)

    @property
    def n_tokens(self) -> int:
        v = self.backbone.vision_tokens
        return sum(s.length(v) for s in self.samples)

    def schemas(self) -> List[dict]:
        """One schema per tenant: the shared-prefix signature plus the
        tenant's output structure."""
        b = self.backbone
        return [dict(backbone_id=b.backbone_id, d_model=b.d,
                     vision_tokens=b.vision_tokens, embed_dtype=0, vocab_id=b.vocab,
                     rope_id=int(b.rope_theta), max_images=t.max_images,
                     action_width=t.width) for t in self.tenants]

    def subset(self, tenants: List[int]) -> "Workload":
        """The same workload restricted to the requests of some tenants, with
        the sample offsets unchanged (they still index the full buffers)."""
        keep = set(tenants)
        w = dataclasses.replace(self, requests=[r for r in self.requests if r.tenant in keep])
        return w


# ---------------------------------------------------------------------------
# workload shapes
# ---------------------------------------------------------------------------

def _interleave(per_tenant: List[List[Sample]], req_batch: int) -> List[Request]:
    """Split each tenant's samples into requests of <= req_batch samples and
    interleave them round-robin across tenants (arrival order)."""
    queues = []
    for t, ss in enumerate(per_tenant):
        queues.append([ss[i:i + req_batch] for i in range(0, len(ss), req_batch)])
    out: List[Request] = []
    k = 0
    while any(k < len(q) for q in queues):
        for t, q in enumerate(queues):
            if k < len(q):
                out.append(Request(tenant=t, schema=t, samples=q[k]))
        k += 1
    return out


def _assign_offsets(w: Workload) -> Workload:
    vrow = tpos = toff = 0
    V = w.backbone.vision_tokens
    for r in w.requests:
        width = w.tenants[r.tenant].width
        for s in r.samples:
            s.vision_row, s.text_pos, s.target_off = vrow, tpos, toff
            vrow += s.n_img * V
            tpos += s.text_len
            toff += width
    return w


def zipf_counts(n_tenants: int, total: int, s: float) -> List[int]:
    """Deterministic Zipf(s) counts over ranks 1..n summing to ``total``: floor
    of the ideal share (at least 1), remainder to the largest fractional parts."""
    ideal = np.array([total * r ** (-s) for r in range(1, n_tenants + 1)])
    ideal = ideal / ideal.sum() * total
    c = np.maximum(1, np.floor(ideal)).astype(int)
    rem = total - int(c.sum())
    frac = ideal - np.floor(ideal)
    order = sorted(range(n_tenants), key=lambda i: (-frac[i], i))
    for i in order[:rem]:
        c[i] += 1
    return [int(x) for x in c]


def make_workload(name: str, **over) -> Workload:
    """Build one of the five named workloads (see the module docstring)."""
    if name == "tiny":
        seed = 0
        bb = Backbone(n_layers=1, d=256, n_heads=4, n_kv_heads=4, head_dim=64, d_ff=1024,
                      vision_tokens=64)
        tenants = [Tenant(HEAD_MLP, chunk=8, action_dim=7, d_hidden=256, max_images=1)
                   for _ in range(2)]
        per = [[Sample(1, 16) for _ in range(4)], [Sample(1, 24) for _ in range(4)]]
        reqs = _interleave(per, 4)
    elif name == "small":
        seed = 1
        rng = np.random.default_rng(seed)
        bb = Backbone(n_layers=6, d=1024, n_heads=16, n_kv_heads=16, head_dim=64, d_ff=4096)
        tenants = [Tenant(HEAD_MLP, chunk=16, action_dim=[7, 14][t % 2], d_hidden=1024,
                          max_images=1) for t in range(8)]
        per = []
        for t in range(8):
            n = int(rng.integers(8, 33))
            per.append([Sample(1, int(rng.integers(8, 49))) for _ in range(n)])
        reqs = _interleave(per, 8)
    elif name in ("mqa2b", "zipf2b"):
        zipf = name == "zipf2b"
        seed = 3 if zipf else 2
        rng = np.random.default_rng(seed)
        bb = Backbone(n_layers=18, d=2048, n_heads=8, n_kv_heads=1, head_dim=256, d_ff=16384,
                      glu=GLU_GEGLU, lora_rank=16 if zipf else 0)
        T = 64 if zipf else 16
        tenants = [Tenant(HEAD_XATTN, chunk=50, action_dim=[7, 14, 32][t % 3], q_dim=256,
                          n_queries=32) for t in range(T)]
        if zipf:
            counts = zipf_counts(T, 512, 1.2)
            perm = rng.permutation(T)
            n_of = [0] * T
            for rank, t in enumerate(perm):
                n_of[int(t)] = counts[rank]
            lo, hi = 4, 72
        else:
            n_of = [16] * T
            lo, hi = 16, 64
        per = [[Sample(1 + t % 3, int(rng.integers(lo, hi + 1))) for _ in range(n_of[t])]
               for t in range(T)]
        reqs = _interleave(per, 8)
    elif name == "llama7b":
        seed = 4
        rng = np.random.default_rng(seed)
        bb = Backbone(n_layers=32, d=4096, n_heads=32, n_kv_heads=32, head_dim=128, d_ff=11008)
        T = 32
        tenants = [Tenant(HEAD_MLP, chunk=8, action_dim=7, d_hidden=1024, max_images=1)
                   for _ in range(T)]
        per: List[List[Sample]] = [[] for _ in range(T)]
        tot, t = 0, 0
        while tot < 65536:
            s = Sample(1, int(rng.integers(16, 65)))
            per[t].append(s)
            tot += s.length(bb.vision_tokens)
            t = (t + 1) % T
        reqs = _interleave(per, 4)
    else:
        raise KeyError(name)
    bb = dataclasses.replace(bb, **{k: v for k, v in over.items() if hasattr(bb, k)})
    w = Workload(name=name, seed=seed, backbone=bb, tenants=tenants, requests=reqs)
    for k, v in over.items():
        if hasattr(w, k) and not hasattr(bb, k):
            setattr(w, k, v)
    return _assign_offsets(w)


WORKLOADS = ("tiny", "small", "mqa2b", "zipf2b", "llama7b")


def custom_workload(backbone: Backbone, tenants: List[Tenant], per_tenant: List[List[Sample]],
                    req_batch: int = 4, seed: int = 0, name: str = "custom",
                    schema_of: Optional[List[int]] = None) -> Workload:
    """A small hand-shaped workload for tests (ragged lengths, odd sizes)."""
    reqs = _interleave(per_tenant, req_batch)
    if schema_of is not None:
        for r in reqs:
            r.schema = schema_of[r.tenant]
    return _assign_offsets(Workload(name=name, seed=seed, backbone=backbone,
                                    tenants=tenants, requests=reqs))


# ---------------------------------------------------------------------------
# tensors
# ---------------------------------------------------------------------------

def _gen(device, seed: int, *key: int):
    import torch
    g = torch.Generator(device=device)
    # a stable per-tensor seed derived from the workload seed and a key
    h = seed * 1000003
    for k in key:
        h = (h * 1000033 + int(k) + 7) % (1 << 62)
    g.manual_seed(h)
    return g


def _normal(shape, std, device, seed, *key, mean=0.0):
    import torch
    g = _gen(device, seed, *key)
    t = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    if mean != 0.0:
        t.add_(mean)
    return t.to(torch.bfloat16)


def make_backbone_weights(w: Workload, device="cpu", std: float = 0.02) -> Dict:
    """Frozen backbone: bf16 N(0, std) projections, bf16 RMSNorm gains 1+N(0, std),
    a shared N(0,1) text-embedding table.  Projections are stored [out, in]."""
    b = w.backbone
    s = w.seed
    qd, kvd = b.n_heads * b.head_dim, b.n_kv_heads * b.head_dim
    layers = []
    for l in range(b.n_layers):
        L = dict(
            attn_norm=_normal((b.d,), std, device, s, 1, l, mean=1.0),
            wq=_normal((qd, b.d), b.qk_std, device, s, 2, l),
            wk=_normal((kvd, b.d), b.qk_std, device, s, 3, l),
            wv=_normal((kvd, b.d), std, device, s, 4, l),
            wo=_normal((b.d, qd), std, device, s, 5, l),
            ffn_norm=_normal((b.d,), std, device, s, 6, l, mean=1.0),
            wg=_normal((b.d_ff, b.d), std, device, s, 7, l),
            wu=_normal((b.d_ff, b.d), std, device, s, 8, l),
            wd=_normal((b.d, b.d_ff), std, device, s, 9, l),
        )
        if b.lora_rank:
            r, T = b.lora_rank, len(w.tenants)
            for j, (nm, din, dout) in enumerate((("q", b.d, qd), ("k", b.d, kvd),
                                                  ("v", b.d, kvd), ("o", qd, b.d))):
                L["lora_a_" + nm] = _normal((T, r, din), std, device, s, 10 + j, l)
                L["lora_b_" + nm] = _normal((T, dout, r), std, device, s, 20 + j, l)
        layers.append(L)
    return dict(layers=layers,
                final_norm=_normal((b.d,), std, device, s, 30, mean=1.0),
                text_table=_normal((b.vocab, b.d), 1.0, device, s, 31))


def make_head_weights(w: Workload, device="cpu", std: float = 0.02) -> List[Dict]:
    """Tenant-private action heads (one slot per tenant), bf16 N(0, std)."""
    b, s = w.backbone, w.seed
    out = []
    for t, tn in enumerate(w.tenants):
        if tn.head_kind == HEAD_MLP:
            out.append(dict(w1=_normal((tn.d_hidden, b.d), std, device, s, 40, t),
                            b1=_normal((tn.d_hidden,), std, device, s, 41, t),
                            w2=_normal((tn.width, tn.d_hidden), std, device, s, 42, t),
                            b2=_normal((tn.width,), std, device, s, 43, t)))
        else:
            nq, dq = tn.n_queries, tn.q_dim
            out.append(dict(q=_normal((nq, dq), std, device, s, 50, t),
                            wk=_normal((dq, b.d), std, device, s, 51, t),
                            wv=_normal((dq, b.d), std, device, s, 52, t),
                            wout=_normal((tn.width, nq * dq), std, device, s, 53, t),
                            bout=_normal((tn.width,), std, device, s, 54, t)))
    return out


def make_flow_weights(n_tenants: int, d_model: int, d_ff: int, n_blocks: int, chunk: int,
                      action_dim: int, d_in: int, seed: int, device="cpu",
                      std: float = 0.02) -> Dict:
    """Flow-matching action experts of n_tenants tenants, stacked over
    tenants: bf16 N(0, std) projections [T, out, in] (the gate and up rows
    of each block separately), N(0, std) biases and positions."""
    T, dm, F = n_tenants, d_model, d_ff
    r = lambda shape, *key: _normal((T,) + shape, std, device, seed, 70, *key)
    out = dict(w_in=r((dm, action_dim), 0), b_in=r((dm,), 1), pos=r((chunk, dm), 2),
               t1=r((dm, dm), 3), tb1=r((dm,), 4), t2=r((dm, dm), 5), tb2=r((dm,), 6),
               w_out=r((action_dim, dm), 7), b_out=r((action_dim,), 8), blocks=[])
    for b in range(n_blocks):
        out["blocks"].append(dict(w_qkv=r((3 * dm, dm), 10, b), w_kvc=r((2 * dm, d_in), 11, b),
                                  w_o=r((dm, dm), 12, b), wg=r((F, dm), 13, b),
                                  wu=r((F, dm), 14, b), w_d=r((dm, F), 15, b)))
    return out


def make_flow_inputs(n_samples: int, chunk: int, action_dim: int, seed: int, device="cpu"):
    """Per sample (packed order): target chunk U(-1, 1), noise N(0, 1), time
    U(0, 1) (the flow-matching draws, made here and passed in)."""
    import torch
    g = _gen(device, seed, 80)
    actions = torch.rand(n_samples, chunk, action_dim, generator=g, device=device) * 2 - 1
    g = _gen(device, seed, 81)
    noise = torch.randn(n_samples, chunk, action_dim, generator=g, device=device)
    g = _gen(device, seed, 82)
    tau = torch.rand(n_samples, generator=g, device=device)
    return dict(actions=actions, noise=noise, tau=tau)


def make_inputs(w: Workload, device="cpu") -> Dict:
    """Per-sample observations: vision rows N(0,1) bf16, text ids uniform in
    [0, vocab) (int32), action targets uniform in (-1, 1) (fp32), all laid out
    in arrival order at the offsets recorded in each Sample."""
    import torch
    b = w.backbone
    nv = max(1, max((s.vision_row + s.n_img * b.vision_tokens for s in w.samples), default=0))
    nt = max(1, max((s.text_pos + s.text_len for s in w.samples), default=0))
    ntg = max(1, max((s.target_off + w.tenants[r.tenant].width
                      for r in w.requests for s in r.samples), default=0))
    vision = _normal((nv, b.d), 1.0, device, w.seed, 60)
    g = _gen(device, w.seed, 61)
    text_ids = torch.randint(0, b.vocab, (nt,), generator=g, device=device, dtype=torch.int32)
    g = _gen(device, w.seed, 62)
    targets = torch.rand(ntg, generator=g, device=device, dtype=torch.float32).mul_(2).sub_(1)
    return dict(vision=vision, text_ids=text_ids, targets=targets)


def bf16_bits(t) -> np.ndarray:
    """A bf16 torch tensor as a numpy uint16 array of its bit patterns."""
    import torch
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def to_numpy_tree(obj):
    """Convert a (nested) dict/list of torch tensors to numpy: bf16 tensors
    become uint16 bit-pattern arrays, everything else plain numpy."""
    import torch
    if isinstance(obj, dict):
        return {k: to_numpy_tree(v) for k, v in obj.items()}
    if isinstance(obj, list):
        return [to_numpy_tree(v) for v in obj]
    if isinstance(obj, torch.Tensor):
        if obj.dtype == torch.bfloat16:
            return bf16_bits(obj)
        return obj.detach().cpu().numpy()
    return obj
