"""The backbone forward in fp64 with the CUDA path's lower-precision storage
points as switches: a test-side diagnostic.

Test infrastructure only.  It is not the oracle, and the product path never
imports it.  It restates the forward of the oracle (pre-norm decoder blocks,
RMSNorm, rotate-half RoPE, within-sample softmax attention, GLU feed-forward,
final RMSNorm; the paper's §5.2 shared backbone under the readings stated in
the oracle's header) in fp64, with one change: it rounds each value the
CUDA path stores or feeds to a tensor-core GEMM in lower precision, at the
same place and to the same format (round to nearest even).  The CUDA path
keeps its residual stream in fp32, reads every GEMM operand in bf16 and
stores several intermediates in bf16.  None of these roundings exists in
the fp64 oracle, so they put a floor under the GPU's distance from the
oracle that no kernel can go below, and this module computes that floor.
With every switch off it computes the oracle's forward; the CPU tests pin
that to 1e-12 of rms.

Rounding points (the switch names):
  norm      the normed rows a projection reads, in bf16.  Where the CUDA
            path folds an RMSNorm into the GEMMs around it, the stored
            operand is bf16(x * gamma) and the product's rows are scaled by
            rsqrt(mean(x^2) + eps) afterwards.  It folds where the residual
            GEMM before the norm has a K loop of at least 4096: the down
            projection (K = F) before the pre-attention norm, and the O
            projection (K = H hd) before the pre-FFN norm.  Elsewhere the
            operand is bf16(x rsqrt(mean(x^2) + eps) gamma).
  qkv       q and k after RoPE, and v, stored in bf16.
  p         the attention probabilities as the P V operand, in bf16,
            relative to the kernel's lazy running max (attention()); the row
            sums use the unrounded values.
  attn_out  the attention output, stored in bf16.
  u         the GLU product act(g) * u, stored in bf16.
  lora_t    the adapter down-projection x A^T, stored in bf16.  Its input is
            the same operand the projection reads; the up-projection adds
            into the projection's accumulator before the row scale.
  resid     the residual stream, rounded to fp32 after every update.
  hidden    the final normed rows handed to a query head, stored in bf16.
  ds        (attention backward) dS = P * (dP - D) in bf16 as the operand
            of dQ = dS K and dK = dS^T Q; there P is the bf16 operand of
            dV = P^T dO, and D = rowsum(dO * O) reads the forward's bf16 O.
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence

import numpy as np

from oracle import model as M

ALL = ("norm", "qkv", "p", "attn_out", "u", "lora_t", "resid", "hidden", "ds")
NONE: tuple = ()


def f32(a: np.ndarray) -> np.ndarray:
    """Round to fp32 (nearest even), returned as float64."""
    return np.asarray(a, dtype=np.float64).astype(np.float32).astype(np.float64)


def bf16(a: np.ndarray) -> np.ndarray:
    """Round to bf16 (nearest even) as the GPU does from an fp32 value:
    first to fp32, then to the 8-bit mantissa.  Returned as float64."""
    f = np.asarray(a, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32)
    # add half an ulp minus one, plus the kept lowest bit (ties to even),
    # then drop the 16 low bits; finite values cannot carry past the sign
    lsb = np.bitwise_and(u, np.uint32(0x10000)).astype(bool)
    u += np.uint32(0x7FFF)
    u += lsb
    u &= np.uint32(0xFFFF0000)
    return f.astype(np.float64)


def folded_norms(bk) -> tuple:
    """(pre-attention norm folded, pre-FFN norm folded) for a backbone with
    fields d_ff, n_heads, head_dim."""
    return bk.d_ff >= 4096, bk.n_heads * bk.head_dim >= 4096


def widen_layer(lw: Dict) -> Dict:
    """One layer's weights widened to float64 once (the bf16 values exactly)."""
    return {k: M.f64(v) for k, v in lw.items()}


class Emulation:
    """The forward over a list of samples, one block at a time.

    bk: the backbone's shape (fields n_heads, n_kv_heads, head_dim, d_ff,
    glu, eps, rope_theta); xs: each sample's embedding rows [L, d];
    tenants: each sample's tenant (selects its adapters); rounding: the
    switches to apply."""

    def __init__(self, bk, xs: Sequence[np.ndarray], tenants: Sequence[int],
                 rounding: Sequence[str] = ALL, folds: Optional[tuple] = None):
        bad = set(rounding) - set(ALL)
        if bad:
            raise ValueError(f"unknown rounding points {sorted(bad)}")
        self.bk = bk
        self.rnd = frozenset(rounding)
        # folds overrides the CUDA path's rule (to pin both forms on small shapes)
        self.fold_attn, self.fold_ffn = folds if folds is not None else folded_norms(bk)
        self.x = [self._r32(np.asarray(x, dtype=np.float64)) for x in xs]
        self.tenants = list(tenants)
        self.lens = [x.shape[0] for x in xs]
        self.cut = np.cumsum([0] + self.lens)

    # -- rounding helpers --------------------------------------------------
    def _bf(self, name, a):
        return bf16(a) if name in self.rnd else a

    def _r32(self, a):
        return f32(a) if "resid" in self.rnd else a

    # -- pieces --------------------------------------------------------------
    def _norm_operand(self, X, gamma, folded):
        """(operand, per-row scale of the product)."""
        r = 1.0 / np.sqrt(np.mean(X * X, axis=1, keepdims=True) + self.bk.eps)
        if folded:
            return self._bf("norm", X * gamma), r
        return self._bf("norm", X * r * gamma), np.ones_like(r)

    def _proj(self, Y, W, scale, lw, name):
        """Y W^T (+ each sample's adapter up-projection), then the row scale."""
        out = Y @ W.T
        if "lora_a_" + name in lw:
            A, B = lw["lora_a_" + name], lw["lora_b_" + name]
            for i, t in enumerate(self.tenants):
                a, b = self.cut[i], self.cut[i + 1]
                tmp = self._bf("lora_t", Y[a:b] @ A[t].T)
                out[a:b] += tmp @ B[t].T
        return out * scale

    def _attention(self, q, k, v, pos):
        """Within one sample: q [L, H, hd], k/v [L, Hkv, hd] -> [L, H hd]."""
        return attention(q, k, v, tuple(r for r in self.rnd if r == "p"))

    # -- one block over every sample ------------------------------------------
    def block(self, lw: Dict) -> None:
        """Apply one decoder block (lw: widened weights) to every sample."""
        bk = self.bk
        H, Hkv, hd = bk.n_heads, bk.n_kv_heads, bk.head_dim
        X = np.concatenate(self.x, axis=0)
        Y, r = self._norm_operand(X, lw["attn_norm"], self.fold_attn)
        q = self._proj(Y, lw["wq"], r, lw, "q")
        k = self._proj(Y, lw["wk"], r, lw, "k")
        v = self._proj(Y, lw["wv"], r, lw, "v")
        outs = []
        for i, L in enumerate(self.lens):
            a, b = self.cut[i], self.cut[i + 1]
            pos = np.arange(L)
            qi = self._bf("qkv", M.rope(q[a:b].reshape(L, H, hd), pos, bk.rope_theta))
            ki = self._bf("qkv", M.rope(k[a:b].reshape(L, Hkv, hd), pos, bk.rope_theta))
            vi = self._bf("qkv", v[a:b].reshape(L, Hkv, hd))
            outs.append(self._bf("attn_out", self._attention(qi, ki, vi, pos)))
        O = np.concatenate(outs, axis=0)
        X = self._r32(X + self._proj(O, lw["wo"], 1.0, lw, "o"))
        Y, r = self._norm_operand(X, lw["ffn_norm"], self.fold_ffn)
        g = (Y @ lw["wg"].T) * r
        u = (Y @ lw["wu"].T) * r
        act = M.silu(g) if bk.glu == 0 else M.gelu_tanh(g)
        Um = self._bf("u", act * u)
        X = self._r32(X + Um @ lw["wd"].T)
        self.x = [X[self.cut[i]:self.cut[i + 1]] for i in range(len(self.lens))]

    def final(self, final_norm) -> List[np.ndarray]:
        """Final RMSNorm rows of every sample (bf16 if the hidden switch is on)."""
        g = M.f64(final_norm)
        out = []
        for x in self.x:
            n = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + self.bk.eps) * g
            out.append(self._bf("hidden", n))
        return out

    def pooled(self, final_norm) -> List[np.ndarray]:
        """Mean-pooled final normed rows (fp32 on the GPU: not rounded here,
        as the hidden switch applies to stored rows only)."""
        g = M.f64(final_norm)
        return [M.mean_pool(x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + self.bk.eps) * g)
                for x in self.x]


def _rounder(rounding):
    return lambda name, a: bf16(a) if name in rounding else a


KEY_TILE = 64    # keys per tile of the forward attention kernel
LAZY_LOG2 = 8.0  # its running max is raised only past this growth (log2 units)


def attention(q, k, v, rounding: Sequence[str] = ALL) -> np.ndarray:
    """One sample's attention (bidirectional, scale 1/sqrt(hd), K/V head
    h // (H / Hkv)) with the rounding points 'p' and 'attn_out'.
    q: [L, H, hd], k/v: [L, Hkv, hd] -> [L, H hd].

    P is formed as the kernel forms it, which decides what its bf16 rounding
    sees: over tiles of KEY_TILE keys, relative to a running max m taken from
    the first tile and raised (with O and the row sum rescaled) only when a
    tile's max exceeds it by more than LAZY_LOG2, so P = 2^(s log2(e) - m)
    can reach 2^8 and the row's largest P is in general not exactly 1; the
    row sum adds the unrounded values.  Without rounding this is the
    softmax of the oracle up to reassociation."""
    rd = _rounder(rounding)
    L, H, hd = q.shape
    grp = H // k.shape[1]
    c = math.log2(math.e) / math.sqrt(hd)
    o = np.empty_like(q)
    for h in range(H):
        g = h // grp
        s = (q[:, h, :] @ k[:, g, :].T) * c
        m = l = O = None
        for k0 in range(0, L, KEY_TILE):
            st = s[:, k0:k0 + KEY_TILE]
            mx = np.max(st, axis=1)
            if m is None:
                m, alpha = mx, np.ones(L)
                l, O = np.zeros(L), np.zeros((L, hd))
            else:
                up = mx > m + LAZY_LOG2
                alpha = np.where(up, np.exp2(m - mx), 1.0)
                m = np.where(up, mx, m)
            p = np.exp2(st - m[:, None])
            O = O * alpha[:, None] + rd("p", p) @ v[k0:k0 + KEY_TILE, g, :]
            l = l * alpha + np.sum(p, axis=1)
        o[:, h, :] = O / l[:, None]
    return rd("attn_out", o.reshape(L, H * hd))


def attention_backward(q, k, v, do, rounding: Sequence[str] = ALL):
    """Gradients of attention() over one sample with the CUDA path's
    backward rounding points ('p', 'ds', and 'attn_out' for the O that D
    reads).  q, do: [L, H, hd]; k, v: [L, Hkv, hd] -> (dq, dk, dv), unrounded
    (the caller applies the output format)."""
    rd = _rounder(rounding)
    L, H, hd = q.shape
    grp = H // k.shape[1]
    sc = 1.0 / math.sqrt(hd)
    dq, dk, dv = np.zeros_like(q), np.zeros_like(k), np.zeros_like(v)
    for h in range(H):
        g = h // grp
        s = q[:, h, :] @ k[:, g, :].T * sc
        e = np.exp(s - np.max(s, axis=1, keepdims=True))
        P = e / np.sum(e, axis=1, keepdims=True)
        O = rd("attn_out", P @ v[:, g, :])
        dv[:, g, :] += rd("p", P).T @ do[:, h, :]
        dP = do[:, h, :] @ v[:, g, :].T
        D = np.sum(do[:, h, :] * O, axis=1, keepdims=True)
        dS = rd("ds", P * (dP - D))
        dq[:, h, :] = dS @ k[:, g, :] * sc
        dk[:, g, :] += dS.T @ q[:, h, :] * sc
    return dq, dk, dv


def forward(bk, weights: Dict, xs: Sequence[np.ndarray], tenants: Sequence[int],
            rounding: Sequence[str] = ALL, n_layers: Optional[int] = None,
            pool: bool = True, folds: Optional[tuple] = None) -> List[np.ndarray]:
    """The whole emulated forward: pooled features (pool) or final rows."""
    em = Emulation(bk, xs, tenants, rounding, folds)
    layers = weights["layers"][: (n_layers if n_layers is not None else len(weights["layers"]))]
    for lw in layers:
        em.block(widen_layer(lw))
    return em.pooled(weights["final_norm"]) if pool else em.final(weights["final_norm"])
