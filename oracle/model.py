"""fp64 definition of the shared backbone forward, tenant heads, loss and grads.

Test infrastructure only (see the package docstring).  Everything is float64;
bf16 weights and inputs arrive as uint16 bit patterns (or any float array)
and are widened exactly.  No blocking, fusion or reordering: each function
is the textbook formula, with numpy's matmul as the only library step.

Where the paper is silent, these readings are taken (the paper fixes only
that a frozen VLM backbone is shared and tenant action modules, losses and
gradients stay private — §3.1, §4.3, §5.2, App. A):

  R1  pre-norm decoder block without biases:
        x <- x + W_o . Attn(RoPE(W_q n1), RoPE(W_k n1), W_v n1),  n1 = RMSNorm(x)
        x <- x + W_d . (act(W_g n2) * (W_u n2)),                 n2 = RMSNorm(x)
      and a final RMSNorm; act = SiLU (SwiGLU) or tanh-GELU (GeGLU).
  R2  RMSNorm(x) = x / sqrt(mean(x^2) + eps) * gamma, eps = 1e-6.
  R3  RoPE, rotate-half pairing (i, i + hd/2), inv_freq_i = theta^(-2i/hd),
      theta = 10000, positions restarting at 0 in every sample.
  R4  attention is bidirectional inside a sample (the observation prefix),
      scale 1/sqrt(hd), no attention across samples; grouped-query sharing
      of K/V heads (query head h uses K/V head h // (H / H_kv)).
  R5  LoRA on Q/K/V/O (when present): y += (x A_t^T) B_t^T with the sample's
      tenant t, scale 1.
  R6  features for an MLP head: the mean over all L_s tokens of the final
      normed hidden; MLP head z = p W1^T + b1, a = SiLU(z), y = a W2^T + b2.
  R7  query head: k = X Wk^T, v = X Wv^T over the sample's final normed
      tokens X; O = softmax(Q k^T / sqrt(dq)) v with the tenant's learned
      queries Q; y = flatten(O) Wout^T + bout.
  R8  per-tenant loss: mean of squared error over the tenant's samples and
      outputs (no 1/2 factor); never summed or averaged across tenants.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np


# ---------------------------------------------------------------------------
# dtype helpers
# ---------------------------------------------------------------------------

def f64(a) -> np.ndarray:
    """Widen to float64; uint16 arrays are bf16 bit patterns (exact)."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return np.asarray(a, dtype=np.float64)


def widen_tree(obj):
    """Widen a nested dict/list of weight arrays to float64 once (for small
    models, so per-sample loops do not re-widen the same weights)."""
    if isinstance(obj, dict):
        return {k: widen_tree(v) for k, v in obj.items()}
    if isinstance(obj, list):
        return [widen_tree(v) for v in obj]
    if isinstance(obj, np.ndarray) and obj.dtype in (np.uint16, np.float32, np.float16):
        return f64(obj)
    return obj


# ---------------------------------------------------------------------------
# elementwise pieces
# ---------------------------------------------------------------------------

def rmsnorm(x: np.ndarray, gamma, eps: float) -> np.ndarray:
    """R2, over the last axis."""
    ms = np.mean(x * x, axis=-1, keepdims=True)
    return x / np.sqrt(ms + eps) * f64(gamma)


def silu(z):
    return z / (1.0 + np.exp(-z))


def silu_grad(z):
    s = 1.0 / (1.0 + np.exp(-z))
    return s * (1.0 + z * (1.0 - s))


def gelu_tanh(z):
    c = math.sqrt(2.0 / math.pi)
    return 0.5 * z * (1.0 + np.tanh(c * (z + 0.044715 * z ** 3)))


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """R3.  x: [L, heads, hd]; pos: [L] integer positions."""
    hd = x.shape[-1]
    half = hd // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / hd)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]  # [L, half]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    lo, hi = x[..., :half], x[..., half:]
    return np.concatenate([lo * c - hi * s, hi * c + lo * s], axis=-1)


def softmax(s: np.ndarray, axis=-1) -> np.ndarray:
    m = np.max(s, axis=axis, keepdims=True)
    e = np.exp(s - m)
    return e / np.sum(e, axis=axis, keepdims=True)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray) -> np.ndarray:
    """R4 over one sample.  q: [L, H, hd], k/v: [L, Hkv, hd] -> [L, H, hd]."""
    L, H, hd = q.shape
    grp = H // k.shape[1]
    out = np.empty_like(q)
    for h in range(H):
        g = h // grp
        p = softmax(q[:, h, :] @ k[:, g, :].T / math.sqrt(hd))
        out[:, h, :] = p @ v[:, g, :]
    return out


# ---------------------------------------------------------------------------
# backbone
# ---------------------------------------------------------------------------

def sample_embeddings(bb: Dict, s: Dict, vision, text_ids, text_table) -> np.ndarray:
    """The sample's own prefix: its vision rows, then its text-token rows."""
    nv = s["n_img"] * bb["vision_tokens"]
    rows = [f64(vision[s["vision_row"]:s["vision_row"] + nv])]
    ids = np.asarray(text_ids[s["text_pos"]:s["text_pos"] + s["text_len"]], dtype=np.int64)
    rows.append(f64(text_table[ids]))
    return np.concatenate(rows, axis=0)


def _proj(x, w, lora_a=None, lora_b=None):
    y = x @ f64(w).T
    if lora_a is not None:
        y = y + (x @ f64(lora_a).T) @ f64(lora_b).T
    return y


def block(bb: Dict, lw: Dict, x: np.ndarray, tenant: int) -> np.ndarray:
    """R1 for one sample's rows x [L, d]."""
    L = x.shape[0]
    H, Hkv, hd = bb["n_heads"], bb["n_kv_heads"], bb["head_dim"]
    lora = "lora_a_q" in lw

    def lo(name):
        if not lora:
            return {}
        return dict(lora_a=lw["lora_a_" + name][tenant], lora_b=lw["lora_b_" + name][tenant])

    n1 = rmsnorm(x, lw["attn_norm"], bb["eps"])
    pos = np.arange(L)
    q = rope(_proj(n1, lw["wq"], **lo("q")).reshape(L, H, hd), pos, bb["rope_theta"])
    k = rope(_proj(n1, lw["wk"], **lo("k")).reshape(L, Hkv, hd), pos, bb["rope_theta"])
    v = _proj(n1, lw["wv"], **lo("v")).reshape(L, Hkv, hd)
    o = attention(q, k, v).reshape(L, H * hd)
    x = x + _proj(o, lw["wo"], **lo("o"))
    n2 = rmsnorm(x, lw["ffn_norm"], bb["eps"])
    gate = n2 @ f64(lw["wg"]).T
    up = n2 @ f64(lw["wu"]).T
    act = silu(gate) if bb["glu"] == 0 else gelu_tanh(gate)
    return x + (act * up) @ f64(lw["wd"]).T


def backbone_sample(bb: Dict, weights: Dict, x: np.ndarray, tenant: int = 0,
                    n_layers: Optional[int] = None) -> np.ndarray:
    """The frozen backbone over one sample alone; returns the final normed
    hidden [L, d]."""
    layers = weights["layers"][: (n_layers if n_layers is not None else len(weights["layers"]))]
    for lw in layers:
        x = block(bb, lw, x, tenant)
    return rmsnorm(x, weights["final_norm"], bb["eps"])


def mean_pool(h: np.ndarray) -> np.ndarray:
    """R6 feature: the mean of a sample's rows."""
    return h.sum(axis=0) / h.shape[0]


# ---------------------------------------------------------------------------
# tenant heads (R6, R7) and loss (R8)
# ---------------------------------------------------------------------------

def mlp_head_forward(hw: Dict, p: np.ndarray):
    """p: [n, d] pooled features of one tenant's samples."""
    z = p @ f64(hw["w1"]).T + f64(hw["b1"])
    a = silu(z)
    y = a @ f64(hw["w2"]).T + f64(hw["b2"])
    return dict(z=z, a=a, y=y)


def mlp_head_backward(hw: Dict, p: np.ndarray, cache: Dict, dy: np.ndarray) -> Dict:
    """Gradients of the loss w.r.t. one tenant's head parameters (no dp: the
    backbone is frozen)."""
    dw2 = dy.T @ cache["a"]
    db2 = dy.sum(axis=0)
    da = dy @ f64(hw["w2"])
    dz = da * silu_grad(cache["z"])
    dw1 = dz.T @ p
    db1 = dz.sum(axis=0)
    return dict(w1=dw1, b1=db1, w2=dw2, b2=db2)


def xattn_head_forward(hw: Dict, X: np.ndarray):
    """X: [L, d] one sample's final normed hidden -> prediction [width]."""
    Q = f64(hw["q"])
    dq = Q.shape[1]
    k = X @ f64(hw["wk"]).T
    v = X @ f64(hw["wv"]).T
    P = softmax(Q @ k.T / math.sqrt(dq))
    O = P @ v
    f = O.reshape(-1)
    y = f @ f64(hw["wout"]).T + f64(hw["bout"])
    return dict(k=k, v=v, P=P, O=O, f=f, y=y)


def xattn_head_backward(hw: Dict, X: np.ndarray, c: Dict, dy: np.ndarray) -> Dict:
    """One sample's contribution to the query head's parameter gradients."""
    Q = f64(hw["q"])
    dq = Q.shape[1]
    sc = 1.0 / math.sqrt(dq)
    dwout = np.outer(dy, c["f"])
    dbout = dy.copy()
    dO = (dy @ f64(hw["wout"])).reshape(c["O"].shape)
    dP = dO @ c["v"].T
    dv = c["P"].T @ dO
    dS = c["P"] * (dP - np.sum(dP * c["P"], axis=1, keepdims=True))
    dQ = dS @ c["k"] * sc
    dk = dS.T @ Q * sc
    return dict(q=dQ, wk=dk.T @ X, wv=dv.T @ X, wout=dwout, bout=dbout)


def l2_loss(y: np.ndarray, t: np.ndarray):
    """R8 for one tenant: y, t [n, width] -> (loss, dloss/dy)."""
    diff = y - f64(t)
    n = diff.size
    return float(np.sum(diff * diff) / n), 2.0 * diff / n


# ---------------------------------------------------------------------------
# the whole grouped step, by its definition
# ---------------------------------------------------------------------------

def backbone_dict(w) -> Dict:
    """Backbone hyper-parameters as a plain dict (from a synth Workload)."""
    b = w.backbone
    return dict(n_heads=b.n_heads, n_kv_heads=b.n_kv_heads, head_dim=b.head_dim, eps=b.eps,
                rope_theta=b.rope_theta, glu=b.glu, vision_tokens=b.vision_tokens, d=b.d)


def sample_features(bb: Dict, weights: Dict, s: Dict, tenant: int, inputs: Dict,
                    head_kind: int, n_layers: Optional[int] = None) -> np.ndarray:
    """Backbone over one sample alone; the pooled feature (MLP head) or the
    final normed hidden rows (query head)."""
    x = sample_embeddings(bb, s, inputs["vision"], inputs["text_ids"], weights["text_table"])
    h = backbone_sample(bb, weights, x, tenant, n_layers)
    return mean_pool(h) if head_kind == 0 else h


def tenant_step(head_kind: int, hw: Dict, feats: List[np.ndarray], targets: np.ndarray):
    """One tenant's head forward, loss and gradients over its samples.

    feats: per sample pooled [d] (MLP) or hidden [L, d] (query head);
    targets: [n, width].  Returns (loss, predictions [n, width], grads)."""
    if head_kind == 0:
        P = np.stack(feats)
        c = mlp_head_forward(hw, P)
        loss, dy = l2_loss(c["y"], targets)
        return loss, c["y"], mlp_head_backward(hw, P, c, dy)
    caches = [xattn_head_forward(hw, X) for X in feats]
    Y = np.stack([c["y"] for c in caches])
    loss, dy = l2_loss(Y, targets)
    grads = None
    for X, c, d in zip(feats, caches, dy):
        g = xattn_head_backward(hw, X, c, d)
        grads = g if grads is None else {k: grads[k] + g[k] for k in g}
    return loss, Y, grads


def grouped_step(w, weights: Dict, heads: List[Dict], inputs: Dict,
                 tenants: Optional[Sequence[int]] = None,
                 n_layers: Optional[int] = None) -> Dict:
    """The grouped path's result by definition: every sample through the
    backbone alone, every tenant's head/loss/grads over its own samples.

    ``w`` is a synth Workload (shapes and offsets only); ``tenants`` limits
    the computation to a subset of whole tenants.  Returns per tenant:
    loss, predictions [n_t, width] (arrival order), grads, features."""
    bb = backbone_dict(w)
    tg = np.asarray(inputs["targets"], dtype=np.float64)
    out = {}
    want = set(range(len(w.tenants)) if tenants is None else tenants)
    for t in sorted(want):
        tn = w.tenants[t]
        samples = [s for r in w.requests if r.tenant == t for s in r.samples]
        if not samples:
            continue
        feats = [sample_features(bb, weights, vars(s), t, inputs, tn.head_kind, n_layers)
                 for s in samples]
        T = np.stack([tg[s.target_off:s.target_off + tn.width] for s in samples])
        loss, Y, grads = tenant_step(tn.head_kind, heads[t], feats, T)
        out[t] = dict(loss=loss, pred=Y, grads=grads, feats=feats)
    return out
