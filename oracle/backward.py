"""fp64 gradients of each tenant's loss with respect to its own LoRA adapters,
back through the frozen shared backbone.

Test infrastructure only (see the package docstring).  It follows the
forward definitions of ``model`` (readings R1-R8 there) and differentiates
them by the chain rule, one sample at a time, with numpy's matmul as the
only library step.

Passages followed:

* §4.3 "Multi-Tenant Group Batching" and §5.2: one shared forward over the
  grouped samples, then tenant-private loss and backward; App. A ("Actor
  Consumption and Version Consistency"): gradients and optimizer state are
  a tenant's own and are never averaged or summed across tenants.
* §3.1: a tenant's trainable action module may be a lightweight adapter
  over the fixed base VLM; §2 places LoRA adapters over one shared base
  among the prior systems.  The adapter's form is reading R5 of ``model``.

Readings where the paper is silent (each a choice, not a statement of the paper):

  L1  the backbone stays frozen: its projections, norms and the text
      embedding table get no gradient; the trainable backbone-side
      parameters are the tenants' LoRA pairs (A_t, B_t) on Q/K/V/O.
  L2  tenant t's adapter gradient is the derivative of tenant t's loss
      alone.  No other tenant's loss depends on (A_t, B_t): samples of
      different tenants never meet inside the backbone (attention stays
      inside a sample, every other step acts per row), so this equals the
      gradient of the sum of all tenants' losses.
  L3  with y = (x A^T) B^T for an adapted projection and gY = dloss/dy:
      dB = gY^T (x A^T), dA = (gY B)^T x, and dloss/dx gains (gY B) A.

Gradients returned per tenant and layer: ``a_q`` [r, d], ``b_q`` [H hd, r],
``a_k``/``a_v`` [r, d], ``b_k``/``b_v`` [Hkv hd, r], ``a_o`` [r, H hd],
``b_o`` [d, r] -- the shapes of one tenant's slice of ``lora_a_*`` /
``lora_b_*``.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import model as M
from .model import f64

PARTS = ("q", "k", "v", "o")


# ---------------------------------------------------------------------------
# elementwise and per-row pieces
# ---------------------------------------------------------------------------

def rmsnorm_backward(x: np.ndarray, gamma, eps: float, dn: np.ndarray) -> np.ndarray:
    """dloss/dx for n = x / sqrt(mean(x^2) + eps) * gamma over the last axis,
    given dn = dloss/dn.  With s = 1/sqrt(mean(x^2) + eps),
    dn_j/dx_i = gamma_j (delta_ij s - x_j x_i s^3 / d)."""
    g = f64(gamma)
    d = x.shape[-1]
    s = 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)
    gdn = dn * g
    return s * gdn - x * s ** 3 * np.sum(gdn * x, axis=-1, keepdims=True) / d


def rope_backward(dy: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """The transpose of R3's rotation: the same pairs rotated by the negative
    angle.  dy: [L, heads, hd]."""
    hd = dy.shape[-1]
    half = hd // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=np.float64) / hd)
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]
    c = np.cos(ang)[:, None, :]
    s = np.sin(ang)[:, None, :]
    lo, hi = dy[..., :half], dy[..., half:]
    return np.concatenate([lo * c + hi * s, hi * c - lo * s], axis=-1)


def gelu_tanh_grad(z):
    c = math.sqrt(2.0 / math.pi)
    t = np.tanh(c * (z + 0.044715 * z ** 3))
    return 0.5 * (1.0 + t) + 0.5 * z * (1.0 - t * t) * c * (1.0 + 3.0 * 0.044715 * z * z)


def attention_backward(q: np.ndarray, k: np.ndarray, v: np.ndarray, do: np.ndarray):
    """Gradients of R4 over one sample.  q, do: [L, H, hd]; k, v: [L, Hkv, hd].
    For query head h on K/V head g:  S = q k^T / sqrt(hd), P = softmax(S),
    dv_g += P^T do_h, dP = do_h v_g^T, dS = P * (dP - rowsum(dP * P)),
    dq_h = dS k_g / sqrt(hd), dk_g += dS^T q_h / sqrt(hd)."""
    L, H, hd = q.shape
    grp = H // k.shape[1]
    sc = 1.0 / math.sqrt(hd)
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for h in range(H):
        g = h // grp
        P = M.softmax(q[:, h, :] @ k[:, g, :].T * sc)
        dv[:, g, :] += P.T @ do[:, h, :]
        dP = do[:, h, :] @ v[:, g, :].T
        dS = P * (dP - np.sum(dP * P, axis=1, keepdims=True))
        dq[:, h, :] = dS @ k[:, g, :] * sc
        dk[:, g, :] += dS.T @ q[:, h, :] * sc
    return dq, dk, dv


# ---------------------------------------------------------------------------
# one block: forward with its intermediates, then backward
# ---------------------------------------------------------------------------

def _lora(lw: Dict, name: str, tenant: int):
    if "lora_a_" + name not in lw:
        return None, None
    return f64(lw["lora_a_" + name][tenant]), f64(lw["lora_b_" + name][tenant])


def block_forward(bb: Dict, lw: Dict, x: np.ndarray, tenant: int):
    """R1 for one sample's rows x [L, d]; returns (output, intermediates)."""
    L = x.shape[0]
    H, Hkv, hd = bb["n_heads"], bb["n_kv_heads"], bb["head_dim"]
    pos = np.arange(L)
    c = dict(x=x, pos=pos)
    n1 = M.rmsnorm(x, lw["attn_norm"], bb["eps"])
    c["n1"] = n1
    pre = {}
    for nm, w, heads in (("q", lw["wq"], H), ("k", lw["wk"], Hkv), ("v", lw["wv"], Hkv)):
        y = n1 @ f64(w).T
        A, B = _lora(lw, nm, tenant)
        if A is not None:
            y = y + (n1 @ A.T) @ B.T
        pre[nm] = y.reshape(L, heads, hd)
    c["q"] = M.rope(pre["q"], pos, bb["rope_theta"])
    c["k"] = M.rope(pre["k"], pos, bb["rope_theta"])
    c["v"] = pre["v"]
    o = M.attention(c["q"], c["k"], c["v"]).reshape(L, H * hd)
    c["o"] = o
    yo = o @ f64(lw["wo"]).T
    A, B = _lora(lw, "o", tenant)
    if A is not None:
        yo = yo + (o @ A.T) @ B.T
    h = x + yo
    c["h"] = h
    n2 = M.rmsnorm(h, lw["ffn_norm"], bb["eps"])
    c["n2"] = n2
    c["gate"] = n2 @ f64(lw["wg"]).T
    c["up"] = n2 @ f64(lw["wu"]).T
    c["act"] = M.silu(c["gate"]) if bb["glu"] == 0 else M.gelu_tanh(c["gate"])
    return h + (c["act"] * c["up"]) @ f64(lw["wd"]).T, c


def _adapter_backward(xin: np.ndarray, gy: np.ndarray, A: np.ndarray, B: np.ndarray):
    """L3 for y = (xin A^T) B^T: returns (dA, dB, contribution to dloss/dxin)."""
    t = xin @ A.T
    gt = gy @ B
    return gt.T @ xin, gy.T @ t, gt @ A


def block_backward(bb: Dict, lw: Dict, c: Dict, dy: np.ndarray, tenant: int):
    """dloss/dx of one block from dy = dloss/d(output), and the adapter
    gradients of the sample's tenant in this block (empty without LoRA)."""
    L = dy.shape[0]
    H, Hkv, hd = bb["n_heads"], bb["n_kv_heads"], bb["head_dim"]
    grads = {}
    # feed-forward sub-block: out = h + (act(gate) * up) Wd^T
    dh = dy.copy()
    dm = dy @ f64(lw["wd"])                      # dloss/d(act * up)
    d_up = dm * c["act"]
    dact = M.silu_grad(c["gate"]) if bb["glu"] == 0 else gelu_tanh_grad(c["gate"])
    d_gate = dm * c["up"] * dact
    dn2 = d_gate @ f64(lw["wg"]) + d_up @ f64(lw["wu"])
    dh = dh + rmsnorm_backward(c["h"], lw["ffn_norm"], bb["eps"], dn2)
    # attention sub-block: h = x + o Wo^T (+ adapter)
    do = dh @ f64(lw["wo"])
    A, B = _lora(lw, "o", tenant)
    if A is not None:
        grads["a_o"], grads["b_o"], extra = _adapter_backward(c["o"], dh, A, B)
        do = do + extra
    dq, dk, dv = attention_backward(c["q"], c["k"], c["v"], do.reshape(L, H, hd))
    gy = dict(q=rope_backward(dq, c["pos"], bb["rope_theta"]).reshape(L, H * hd),
              k=rope_backward(dk, c["pos"], bb["rope_theta"]).reshape(L, Hkv * hd),
              v=dv.reshape(L, Hkv * hd))
    dn1 = gy["q"] @ f64(lw["wq"]) + gy["k"] @ f64(lw["wk"]) + gy["v"] @ f64(lw["wv"])
    for nm in ("q", "k", "v"):
        A, B = _lora(lw, nm, tenant)
        if A is not None:
            grads["a_" + nm], grads["b_" + nm], extra = _adapter_backward(c["n1"], gy[nm], A, B)
            dn1 = dn1 + extra
    dx = dh + rmsnorm_backward(c["x"], lw["attn_norm"], bb["eps"], dn1)
    return dx, grads


# ---------------------------------------------------------------------------
# heads: dloss/d(feature)
# ---------------------------------------------------------------------------

def head_feature_grads(head_kind: int, hw: Dict, feats: List[np.ndarray],
                       targets: np.ndarray) -> List[np.ndarray]:
    """dloss_t/d(feature) for each of the tenant's samples: the pooled
    feature [d] for an MLP head (R6), the final normed rows [L, d] for a
    query head (R7)."""
    if head_kind == 0:
        P = np.stack(feats)
        c = M.mlp_head_forward(hw, P)
        _, dy = M.l2_loss(c["y"], targets)
        dz = (dy @ f64(hw["w2"])) * M.silu_grad(c["z"])
        return list(dz @ f64(hw["w1"]))
    caches = [M.xattn_head_forward(hw, X) for X in feats]
    _, dy = M.l2_loss(np.stack([c["y"] for c in caches]), targets)
    Q = f64(hw["q"])
    sc = 1.0 / math.sqrt(Q.shape[1])
    out = []
    for c, d in zip(caches, dy):
        dO = (d @ f64(hw["wout"])).reshape(c["O"].shape)
        dP = dO @ c["v"].T
        dS = c["P"] * (dP - np.sum(dP * c["P"], axis=1, keepdims=True))
        dk = dS.T @ Q * sc
        dv = c["P"].T @ dO
        out.append(dk @ f64(hw["wk"]) + dv @ f64(hw["wv"]))
    return out


# ---------------------------------------------------------------------------
# the whole path
# ---------------------------------------------------------------------------

def sample_forward(bb: Dict, weights: Dict, x: np.ndarray, tenant: int,
                   n_layers: Optional[int] = None):
    """Backbone over one sample, keeping every block's intermediates.
    Returns (final residual x_L, final normed rows, caches)."""
    layers = weights["layers"][: (n_layers if n_layers is not None else len(weights["layers"]))]
    caches = []
    for lw in layers:
        x, c = block_forward(bb, lw, x, tenant)
        caches.append(c)
    return x, M.rmsnorm(x, weights["final_norm"], bb["eps"]), caches


def sample_backward(bb: Dict, weights: Dict, xL: np.ndarray, caches: List[Dict],
                    d_hidden: np.ndarray, tenant: int):
    """From dloss/d(final normed rows) back to every block; returns the
    per-layer adapter gradients and dloss/d(embedded rows)."""
    dx = rmsnorm_backward(xL, weights["final_norm"], bb["eps"], d_hidden)
    grads: List[Dict] = [None] * len(caches)
    for l in range(len(caches) - 1, -1, -1):
        dx, grads[l] = block_backward(bb, weights["layers"][l], caches[l], dx, tenant)
    return grads, dx


def lora_step(w, weights: Dict, heads: List[Dict], inputs: Dict,
              tenants: Optional[Sequence[int]] = None,
              n_layers: Optional[int] = None) -> Dict:
    """Per tenant: loss, predictions, head gradients (as ``model``), the
    gradient of the loss with respect to each sample's final normed rows
    (``d_hidden``, [L_s, d] per sample in arrival order) and the adapter
    gradients of every layer (``lora``, summed over the tenant's samples)."""
    bb = M.backbone_dict(w)
    tg = np.asarray(inputs["targets"], dtype=np.float64)
    out = {}
    want = set(range(len(w.tenants)) if tenants is None else tenants)
    for t in sorted(want):
        tn = w.tenants[t]
        samples = [s for r in w.requests if r.tenant == t for s in r.samples]
        if not samples:
            continue
        fw = []
        for s in samples:
            x0 = M.sample_embeddings(bb, vars(s), inputs["vision"], inputs["text_ids"],
                                     weights["text_table"])
            fw.append(sample_forward(bb, weights, x0, t, n_layers))
        feats = [M.mean_pool(hn) if tn.head_kind == 0 else hn for _, hn, _ in fw]
        T = np.stack([tg[s.target_off:s.target_off + tn.width] for s in samples])
        loss, Y, hgrads = M.tenant_step(tn.head_kind, heads[t], feats, T)
        dfeat = head_feature_grads(tn.head_kind, heads[t], feats, T)
        lora = None
        d_hidden = []
        for (xL, hn, caches), df in zip(fw, dfeat):
            dh = np.tile(df / hn.shape[0], (hn.shape[0], 1)) if tn.head_kind == 0 else df
            d_hidden.append(dh)
            g, _ = sample_backward(bb, weights, xL, caches, dh, t)
            lora = g if lora is None else [{k: a[k] + b[k] for k in a} for a, b in zip(lora, g)]
        out[t] = dict(loss=loss, pred=Y, grads=hgrads, d_hidden=d_hidden, lora=lora)
    return out
