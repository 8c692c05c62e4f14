"""fp64 flow-matching action expert (a DiT head) as a tenant's private module:
forward, loss and the gradients of the loss with respect to its parameters.

Test infrastructure only (see the package docstring).  numpy matmul is the
only library step; no blocking, fusion or reordering.

Passages followed:

* §3.1: the action module that maps the backbone's latent representation to
  robot actions can be a diffusion or flow-matching action expert, a
  lightweight MLP or a projection head; it is the tenant-specific part.
* §5.2: QwenGR00T decodes with a GR00T-style flow-matching action head over
  the Qwen VLM's features, pi-0.5 is similar in design; the action head is
  the tenant-private module, the VLM the resident base; even a large DiT
  action head costs less than the base VLM's forward.

The paper prints no equation of the expert.  Readings (each a choice, not a statement of the paper):

  F1  rectified-flow training: with the tenant's target chunk a [C, D],
      noise eps [C, D] and time tau in [0, 1] per sample (drawn by the
      caller and passed in), x = tau a + (1 - tau) eps, the target velocity
      is u = a - eps and the loss is the mean of (v - u)^2 over the tenant's
      samples and chunk elements (never mixed across tenants, as R8).
  F2  time embedding: s(tau)_i = sin(1000 tau w_i) for i < dm/2 and
      cos(1000 tau w_(i - dm/2)) after, w_i = 10000^(-i / (dm/2));
      phi = T2 SiLU(T1 s + tb1) + tb2.
  F3  token embedding: h = x W_in^T + b_in + pos + phi (pos [C, dm] learned).
  F4  blocks, pre-norm with non-affine RMSNorm n(h) = h / sqrt(mean(h^2)
      + 1e-6):
        q | k_a | v_a = n(h) W_qkv^T,  k_c | v_c = X W_kvc^T  (X: the
        sample's final normed backbone rows [L, d]),
        per head (width dm / n_heads): softmax(q [k_c; k_a]^T / sqrt(hd))
        [v_c; v_a] -- the action tokens attend to the sample's context
        rows and to each other, bidirectionally;
        h += o W_o^T;  h += (SiLU(n(h) W_g^T) * (n(h) W_u^T)) W_d^T.
  F5  velocity v = n(h) W_out^T + b_out [C, D].
  F6  the backbone stays frozen: no gradient reaches X.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import model as M
from .model import f64

EPS = 1e-6


def norm(h):
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + EPS)


def norm_backward(h, dn):
    """Gradient of the non-affine RMSNorm (the affine one with gamma = 1)."""
    d = h.shape[-1]
    s = 1.0 / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + EPS)
    return s * dn - h * s ** 3 * np.sum(dn * h, axis=-1, keepdims=True) / d


def time_features(tau: float, dm: int) -> np.ndarray:
    """F2: sinusoidal features of 1000 tau."""
    half = dm // 2
    w = 10000.0 ** (-np.arange(half, dtype=np.float64) / half)
    a = 1000.0 * float(tau) * w
    return np.concatenate([np.sin(a), np.cos(a)])


def _attn(q, k, v, nh):
    """Multi-head softmax attention (no mask); returns output and probabilities."""
    C, dm = q.shape
    hd = dm // nh
    out = np.zeros_like(q)
    Ps = []
    for j in range(nh):
        sl = slice(j * hd, (j + 1) * hd)
        P = M.softmax(q[:, sl] @ k[:, sl].T / math.sqrt(hd))
        out[:, sl] = P @ v[:, sl]
        Ps.append(P)
    return out, Ps


def forward(p: Dict, nh: int, X: np.ndarray, a: np.ndarray, eps: np.ndarray, tau: float):
    """One training sample (F1): returns the velocity [C, D], the target u
    and the intermediates the backward reads."""
    a, eps = f64(a), f64(eps)
    v, c = network(p, nh, X, tau * a + (1.0 - tau) * eps, tau)
    return v, a - eps, c


def network(p: Dict, nh: int, X: np.ndarray, x: np.ndarray, tau: float):
    """F2-F5: the velocity v(x, tau) [C, D] of the chunk x given the
    sample's context rows X, and the intermediates."""
    W = {k: f64(v) if not isinstance(v, list) else v for k, v in p.items()}
    dm = W["w_in"].shape[0]
    x = f64(x)
    s = time_features(tau, dm)
    z1 = W["t1"] @ s + W["tb1"]
    phi = W["t2"] @ M.silu(z1) + W["tb2"]
    h = x @ W["w_in"].T + W["b_in"] + W["pos"] + phi
    c = dict(x=x, s=s, z1=z1, blocks=[])
    for B in W["blocks"]:
        B = {k: f64(v) for k, v in B.items()}
        bc = dict(h_in=h)
        n1 = norm(h)
        qkv = n1 @ B["wqkv"].T
        q, ka, va = np.split(qkv, 3, axis=1)
        kvc = X @ B["wkvc"].T
        kc, vc = np.split(kvc, 2, axis=1)
        K, V = np.concatenate([kc, ka]), np.concatenate([vc, va])
        o, Ps = _attn(q, K, V, nh)
        h = h + o @ B["wo"].T
        bc.update(n1=n1, q=q, K=K, V=V, Ps=Ps, o=o, h_mid=h)
        n2 = norm(h)
        g, up = n2 @ B["wg"].T, n2 @ B["wu"].T
        m = M.silu(g) * up
        h = h + m @ B["wd"].T
        bc.update(n2=n2, g=g, up=up, m=m)
        c["blocks"].append(bc)
    c["h_out"] = h
    nf = norm(h)
    c["nf"] = nf
    return nf @ W["w_out"].T + W["b_out"], c


def backward(p: Dict, nh: int, X: np.ndarray, c: Dict, dv: np.ndarray) -> Dict:
    """Gradients of a loss with dloss/dv = dv for one sample."""
    W = {k: f64(v) if not isinstance(v, list) else v for k, v in p.items()}
    dm = W["w_in"].shape[0]
    hd = dm // nh
    g = {}
    g["w_out"] = dv.T @ c["nf"]
    g["b_out"] = dv.sum(axis=0)
    dh = norm_backward(c["h_out"], dv @ W["w_out"])
    gb: List[Dict] = [None] * len(W["blocks"])
    for b in range(len(W["blocks"]) - 1, -1, -1):
        B = {k: f64(v) for k, v in W["blocks"][b].items()}
        bc = c["blocks"][b]
        G = {}
        # MLP: h += (SiLU(g) * up) W_d^T
        G["wd"] = dh.T @ bc["m"]
        dmm = dh @ B["wd"]
        dg = dmm * bc["up"] * M.silu_grad(bc["g"])
        dup = dmm * M.silu(bc["g"])
        G["wg"] = dg.T @ bc["n2"]
        G["wu"] = dup.T @ bc["n2"]
        dh = dh + norm_backward(bc["h_mid"], dg @ B["wg"] + dup @ B["wu"])
        # attention: h += o W_o^T
        G["wo"] = dh.T @ bc["o"]
        do = dh @ B["wo"]
        dq = np.zeros_like(bc["q"])
        dK = np.zeros_like(bc["K"])
        dV = np.zeros_like(bc["V"])
        for j in range(nh):
            sl = slice(j * hd, (j + 1) * hd)
            P = bc["Ps"][j]
            dV[:, sl] = P.T @ do[:, sl]
            dP = do[:, sl] @ bc["V"][:, sl].T
            dS = P * (dP - np.sum(dP * P, axis=1, keepdims=True))
            dq[:, sl] = dS @ bc["K"][:, sl] / math.sqrt(hd)
            dK[:, sl] = dS.T @ bc["q"][:, sl] / math.sqrt(hd)
        L = X.shape[0]
        dqkv = np.concatenate([dq, dK[L:], dV[L:]], axis=1)
        G["wqkv"] = dqkv.T @ bc["n1"]
        G["wkvc"] = np.concatenate([dK[:L], dV[:L]], axis=1).T @ X
        dh = dh + norm_backward(bc["h_in"], dqkv @ B["wqkv"])
        gb[b] = G
    g["blocks"] = gb
    # embedding: h = x W_in^T + b_in + pos + phi
    g["w_in"] = dh.T @ c["x"]
    g["b_in"] = dh.sum(axis=0)
    g["pos"] = dh.copy()
    dphi = dh.sum(axis=0)
    g["t2"] = np.outer(dphi, M.silu(c["z1"]))
    g["tb2"] = dphi
    dz1 = (dphi @ W["t2"]) * M.silu_grad(c["z1"])
    g["t1"] = np.outer(dz1, c["s"])
    g["tb1"] = dz1
    return g


def _add(a, b):
    if a is None:
        return b
    out = {k: a[k] + b[k] for k in a if k != "blocks"}
    out["blocks"] = [{k: x[k] + y[k] for k in x} for x, y in zip(a["blocks"], b["blocks"])]
    return out


def tenant_step(p: Dict, nh: int, contexts: List[np.ndarray], acts: np.ndarray,
                noise: np.ndarray, taus: Sequence[float]):
    """F1 over one tenant's samples: (loss, velocities [n, C, D], gradients)."""
    outs = [forward(p, nh, X, a, e, t) for X, a, e, t in zip(contexts, acts, noise, taus)]
    V = np.stack([o[0] for o in outs])
    U = np.stack([o[1] for o in outs])
    diff = V - U
    loss = float(np.sum(diff * diff) / diff.size)
    dV = 2.0 * diff / diff.size
    grads = None
    for (v, u, c), X, dv in zip(outs, contexts, dV):
        grads = _add(grads, backward(p, nh, X, c, dv))
    return loss, V, grads


def sample(p: Dict, nh: int, X: np.ndarray, noise: np.ndarray, n_steps: int) -> np.ndarray:
    """Inference: integrate dx/dtau = v(x, tau) from tau = 0 (x = the noise)
    to tau = 1 with n_steps Euler steps (the forward of F3-F5 at each)."""
    x = f64(noise).copy()
    dt = 1.0 / n_steps
    for i in range(n_steps):
        v, _ = network(p, nh, X, x, i * dt)
        x = x + dt * v
    return x
