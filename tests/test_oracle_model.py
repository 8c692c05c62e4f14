"""Pins for the oracle's backbone, heads, loss and gradients (CPU only).

Each pin is independent of the oracle's own formulas: hand values, closed
forms, special cases that reduce to a textbook result, brute force with
explicit loops, central finite differences, and the invariants the method
must keep (grouped == isolated, slot isolation)."""
import math

import numpy as np
import pytest

import synth
from oracle import model as M
from oracle import plan as P
from tests.helpers import oracle_requests

RNG = np.random.default_rng(123)


# ---------------- RMSNorm ----------------------------------------------------

def test_rmsnorm_hand_values():
    x = np.array([[3.0, 4.0]])
    np.testing.assert_allclose(M.rmsnorm(x, np.ones(2), 0.0), x / math.sqrt(12.5), rtol=1e-15)
    c = np.full((1, 8), 2.5)
    g = np.linspace(0.5, 1.5, 8)
    np.testing.assert_allclose(M.rmsnorm(c, g, 1e-6)[0], g * 2.5 / math.sqrt(6.25 + 1e-6), rtol=1e-14)
    # scale invariance when eps = 0
    y = RNG.standard_normal((3, 16))
    np.testing.assert_allclose(M.rmsnorm(7.0 * y, np.ones(16), 0.0), M.rmsnorm(y, np.ones(16), 0.0),
                               rtol=1e-13)


def test_bf16_widening_is_exact():
    bits = np.array([0x3F80, 0xC000, 0x3E80, 0x0000, 0x7F7F], dtype=np.uint16)
    np.testing.assert_array_equal(M.f64(bits), [1.0, -2.0, 0.25, 0.0, 3.3895313892515355e38])


# ---------------- RoPE -------------------------------------------------------

def test_rope_hand_values():
    x = np.zeros((1, 1, 4))
    x[0, 0, 0] = 1.0
    y = M.rope(x, np.array([1]), 10000.0)
    np.testing.assert_allclose(y[0, 0], [math.cos(1), 0, math.sin(1), 0], atol=1e-15)
    x = np.zeros((1, 1, 4))
    x[0, 0, 1] = 1.0   # second pair rotates at 10000^(-2/4) = 0.01 rad per position
    y = M.rope(x, np.array([3]), 10000.0)
    np.testing.assert_allclose(y[0, 0], [0, math.cos(0.03), 0, math.sin(0.03)], atol=1e-15)


def test_rope_identity_at_zero_norm_and_relative_position():
    x = RNG.standard_normal((5, 3, 64))
    np.testing.assert_array_equal(M.rope(x[:1], np.array([0]), 1e4), x[:1])
    y = M.rope(x, np.arange(5) * 37, 1e4)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    q, k = RNG.standard_normal((1, 1, 64)), RNG.standard_normal((1, 1, 64))
    d1 = (M.rope(q, [10], 1e4) * M.rope(k, [3], 1e4)).sum()
    d2 = (M.rope(q, [107], 1e4) * M.rope(k, [100], 1e4)).sum()
    assert abs(d1 - d2) < 1e-10


# ---------------- activations -----------------------------------------------

def test_activation_special_values():
    assert M.silu(0.0) == 0.0 and abs(M.silu(40.0) - 40.0) < 1e-12
    assert abs(M.silu_grad(0.0) - 0.5) < 1e-15
    z = np.linspace(-6, 6, 101)
    h = 1e-6
    np.testing.assert_allclose(M.silu_grad(z), (M.silu(z + h) - M.silu(z - h)) / (2 * h), atol=1e-9)
    # tanh GELU is within 1e-3 of the exact erf GELU (textbook approximation)
    exact = np.array([0.5 * v * (1 + math.erf(v / math.sqrt(2))) for v in z])
    assert np.max(np.abs(M.gelu_tanh(z) - exact)) < 1e-3
    assert M.gelu_tanh(0.0) == 0.0


# ---------------- attention --------------------------------------------------

def test_attention_special_cases():
    v = RNG.standard_normal((1, 2, 8))
    q = RNG.standard_normal((1, 2, 8))
    np.testing.assert_allclose(M.attention(q, RNG.standard_normal((1, 2, 8)), v), v)   # L = 1
    L = 6
    v = RNG.standard_normal((L, 2, 8))
    out = M.attention(np.zeros((L, 2, 8)), RNG.standard_normal((L, 2, 8)), v)
    np.testing.assert_allclose(out, np.broadcast_to(v.mean(axis=0), out.shape), rtol=1e-13)
    # a query aligned with one of several orthogonal keys picks that key's value
    k = np.zeros((4, 1, 8))
    for j in range(4):
        k[j, 0, j] = 1.0
    q = np.zeros((4, 1, 8))
    for i in range(4):
        q[i, 0, 3 - i] = 1e3
    v = RNG.standard_normal((4, 1, 8))
    np.testing.assert_allclose(M.attention(q, k, v)[:, 0], v[::-1, 0], atol=1e-12)


def test_attention_brute_force_and_kv_groups():
    L, H, Hkv, hd = 5, 4, 2, 6
    q, k, v = (RNG.standard_normal((L, h, hd)) for h in (H, Hkv, Hkv))
    out = M.attention(q, k, v)
    for h in range(H):
        g = h // 2
        for i in range(L):
            s = [sum(q[i, h, c] * k[j, g, c] for c in range(hd)) / math.sqrt(hd) for j in range(L)]
            e = [math.exp(x - max(s)) for x in s]
            ref = [sum(e[j] * v[j, g, c] for j in range(L)) / sum(e) for c in range(hd)]
            np.testing.assert_allclose(out[i, h], ref, rtol=1e-12)
    v2 = v.copy()
    v2[:, 1] = 0.0   # kv head 1 serves query heads 2 and 3 only
    o2 = M.attention(q, k, v2)
    assert np.all(o2[:, 2:] == 0) and np.allclose(o2[:, :2], out[:, :2])


# ---------------- backbone structure -----------------------------------------

def _tiny_bb(**kw):
    base = dict(n_heads=2, n_kv_heads=1, head_dim=8, eps=1e-6, rope_theta=1e4, glu=0,
                vision_tokens=2, d=16)
    base.update(kw)
    return base


def _layer(d=16, H=2, Hkv=1, hd=8, F=24, scale=0.3):
    return dict(attn_norm=1 + 0.1 * RNG.standard_normal(d),
                wq=scale * RNG.standard_normal((H * hd, d)),
                wk=scale * RNG.standard_normal((Hkv * hd, d)),
                wv=scale * RNG.standard_normal((Hkv * hd, d)),
                wo=scale * RNG.standard_normal((d, H * hd)),
                ffn_norm=1 + 0.1 * RNG.standard_normal(d),
                wg=scale * RNG.standard_normal((F, d)), wu=scale * RNG.standard_normal((F, d)),
                wd=scale * RNG.standard_normal((d, F)))


def test_block_with_zero_output_projections_is_identity():
    lw = _layer()
    lw["wo"][:] = 0
    lw["wd"][:] = 0
    x = RNG.standard_normal((7, 16))
    np.testing.assert_array_equal(M.block(_tiny_bb(), lw, x, 0), x)


def test_block_single_token_reduces_to_value_path():
    # L = 1: attention returns v and RoPE at position 0 is the identity, so the
    # block is x + Wo Wv n1 followed by the FFN on the updated stream.
    lw = _layer()
    bb = _tiny_bb()
    x = RNG.standard_normal((1, 16))
    n1 = x / np.sqrt(np.mean(x * x) + 1e-6) * lw["attn_norm"]
    vrow = lw["wv"] @ n1[0]
    h = x[0] + lw["wo"] @ np.concatenate([vrow, vrow])   # both query heads share kv head 0
    n2 = h / np.sqrt(np.mean(h * h) + 1e-6) * lw["ffn_norm"]
    g, u = lw["wg"] @ n2, lw["wu"] @ n2
    ref = h + lw["wd"] @ (g / (1 + np.exp(-g)) * u)
    np.testing.assert_allclose(M.block(bb, lw, x, 0)[0], ref, rtol=1e-12)


def test_lora_adds_low_rank_update():
    lw = _layer()
    x = RNG.standard_normal((3, 16))
    base = M.block(_tiny_bb(), lw, x, 0)
    for nm, din, dout in (("q", 16, 16), ("k", 16, 8), ("v", 16, 8), ("o", 16, 16)):
        lw["lora_a_" + nm] = np.zeros((2, 4, din))
        lw["lora_b_" + nm] = RNG.standard_normal((2, dout, 4))
    np.testing.assert_allclose(M.block(_tiny_bb(), lw, x, 1), base, rtol=1e-13)  # A = 0
    lw["lora_a_v"] = RNG.standard_normal((2, 4, 16))
    assert not np.allclose(M.block(_tiny_bb(), lw, x, 1), base)


def test_mean_pool_constant_rows():
    r = RNG.standard_normal(9)
    np.testing.assert_allclose(M.mean_pool(np.tile(r, (5, 1))), r, rtol=1e-15)


# ---------------- heads, loss, gradients -------------------------------------

def _mlp_head(d=12, dh=10, width=6):
    return dict(w1=0.3 * RNG.standard_normal((dh, d)), b1=0.1 * RNG.standard_normal(dh),
                w2=0.3 * RNG.standard_normal((width, dh)), b2=0.1 * RNG.standard_normal(width))


def _xattn_head(d=12, nq=3, dq=4, width=5):
    return dict(q=RNG.standard_normal((nq, dq)), wk=0.5 * RNG.standard_normal((dq, d)),
                wv=0.5 * RNG.standard_normal((dq, d)),
                wout=0.3 * RNG.standard_normal((width, nq * dq)),
                bout=0.1 * RNG.standard_normal(width))


def _fd_check(kind, hw, feats, T):
    loss, _, grads = M.tenant_step(kind, hw, feats, T)
    h = 1e-6
    for name, g in grads.items():
        flat = hw[name].reshape(-1)
        for idx in RNG.choice(flat.size, size=min(flat.size, 12), replace=False):
            old = flat[idx]
            flat[idx] = old + h
            lp = M.tenant_step(kind, hw, feats, T)[0]
            flat[idx] = old - h
            lm = M.tenant_step(kind, hw, feats, T)[0]
            flat[idx] = old
            fd = (lp - lm) / (2 * h)
            an = g.reshape(-1)[idx]
            assert abs(fd - an) <= 1e-6 * max(1.0, abs(fd)) + 1e-9, (name, idx, fd, an)


def test_mlp_head_gradients_finite_differences():
    hw = _mlp_head()
    feats = [RNG.standard_normal(12) for _ in range(4)]
    _fd_check(0, hw, feats, RNG.uniform(-1, 1, (4, 6)))


def test_xattn_head_gradients_finite_differences():
    hw = _xattn_head()
    feats = [RNG.standard_normal((L, 12)) for L in (1, 3, 7)]
    _fd_check(1, hw, feats, RNG.uniform(-1, 1, (3, 5)))


def test_loss_closed_form_and_zero_gradient_case():
    t = RNG.uniform(-1, 1, (3, 4))
    loss, dy = M.l2_loss(t + 0.25, t)
    assert abs(loss - 0.0625) < 1e-15
    np.testing.assert_allclose(dy, np.full((3, 4), 2 * 0.25 / 12))
    hw = _mlp_head(width=4)
    hw["w2"][:] = 0
    T = np.tile(hw["b2"], (3, 1))
    loss, y, g = M.tenant_step(0, hw, [RNG.standard_normal(12) for _ in range(3)], T)
    assert loss == 0.0 and all(np.all(v == 0) for v in g.values())


def test_xattn_head_single_token_is_linear_in_value():
    # one key: the softmax is 1, every query reads v = Wv x
    hw = _xattn_head()
    X = RNG.standard_normal((1, 12))
    c = M.xattn_head_forward(hw, X)
    v = hw["wv"] @ X[0]
    np.testing.assert_allclose(c["O"], np.tile(v, (3, 1)), rtol=1e-13)


# ---------------- whole path: grouped == isolated, slot isolation -------------

def _small_custom():
    bb = synth.Backbone(n_layers=2, d=32, n_heads=2, n_kv_heads=1, head_dim=16, d_ff=48,
                        vision_tokens=4, vocab=50, qk_std=0.2)
    tenants = [synth.Tenant(synth.HEAD_MLP, chunk=2, action_dim=3, d_hidden=16, max_images=2),
               synth.Tenant(synth.HEAD_XATTN, chunk=2, action_dim=2, n_queries=3, q_dim=8,
                            max_images=2),
               synth.Tenant(synth.HEAD_MLP, chunk=1, action_dim=5, d_hidden=8, max_images=2)]
    per = [[synth.Sample(1, 3), synth.Sample(0, 5)], [synth.Sample(2, 1)],
           [synth.Sample(1, 0), synth.Sample(2, 2), synth.Sample(0, 1)]]
    return synth.custom_workload(bb, tenants, per, req_batch=1, seed=9)


def _tensors(w):
    wt = synth.to_numpy_tree(synth.make_backbone_weights(w, std=0.2))
    hd = synth.to_numpy_tree(synth.make_head_weights(w, std=0.2))
    inp = synth.to_numpy_tree(synth.make_inputs(w))
    return wt, hd, inp


def _packed_forward(w, wt, inp):
    """Test-side packed formulation: all accepted samples in one sequence with
    a block-diagonal mask built from the plan, positions from the plan.  Must
    agree with the oracle's per-sample definition."""
    b = w.backbone
    p = P.group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    src = np.array(p["gather_src"])
    X = np.where((src >= 0)[:, None], M.f64(inp["vision"][np.maximum(src, 0)]),
                 M.f64(wt["text_table"][inp["text_ids"][np.maximum(-src - 1, 0)]]))
    cu = p["cu_seqlens"]
    N = X.shape[0]
    seg = np.zeros(N, dtype=int)
    for i in range(len(cu) - 1):
        seg[cu[i]:cu[i + 1]] = i
    mask = seg[:, None] == seg[None, :]
    pos = np.array(p["pos_ids"])
    H, Hkv, hd = b.n_heads, b.n_kv_heads, b.head_dim
    for lw in wt["layers"]:
        n1 = M.rmsnorm(X, lw["attn_norm"], b.eps)
        q = M.rope((n1 @ M.f64(lw["wq"]).T).reshape(N, H, hd), pos, b.rope_theta)
        k = M.rope((n1 @ M.f64(lw["wk"]).T).reshape(N, Hkv, hd), pos, b.rope_theta)
        v = (n1 @ M.f64(lw["wv"]).T).reshape(N, Hkv, hd)
        o = np.empty((N, H, hd))
        for h in range(H):
            s = q[:, h] @ k[:, h // (H // Hkv)].T / math.sqrt(hd)
            s = np.where(mask, s, -np.inf)
            e = np.exp(s - s.max(axis=1, keepdims=True))
            o[:, h] = (e / e.sum(axis=1, keepdims=True)) @ v[:, h // (H // Hkv)]
        X = X + o.reshape(N, H * hd) @ M.f64(lw["wo"]).T
        n2 = M.rmsnorm(X, lw["ffn_norm"], b.eps)
        X = X + (M.silu(n2 @ M.f64(lw["wg"]).T) * (n2 @ M.f64(lw["wu"]).T)) @ M.f64(lw["wd"]).T
    return p, M.rmsnorm(X, wt["final_norm"], b.eps)


def test_packed_varlen_equals_isolated_samples():
    w = _small_custom()
    wt, hd, inp = _tensors(w)
    p, Hp = _packed_forward(w, wt, inp)
    bb = M.backbone_dict(w)
    acc = [s for r in w.requests for s in r.samples]
    # packed sample i is the i-th sample in slot order; rebuild that order
    order = [s for t in p["slot_tenant"] for r in w.requests if r.tenant == t for s in r.samples]
    assert len(order) == len(acc)
    for i, s in enumerate(order):
        x = M.sample_embeddings(bb, vars(s), inp["vision"], inp["text_ids"], wt["text_table"])
        h = M.backbone_sample(bb, wt, x)
        np.testing.assert_allclose(Hp[p["cu_seqlens"][i]:p["cu_seqlens"][i + 1]], h,
                                   rtol=1e-10, atol=1e-12)


def test_grouped_step_equals_isolated_tenant_steps_and_isolates_slots():
    w = _small_custom()
    wt, hd, inp = _tensors(w)
    full = M.grouped_step(w, wt, hd, inp)
    for t in range(3):
        iso = M.grouped_step(w.subset([t]), wt, hd, inp)[t]
        assert iso["loss"] == full[t]["loss"]
        for k in iso["grads"]:
            np.testing.assert_array_equal(iso["grads"][k], full[t]["grads"][k])
    # perturbing tenant 0's targets changes nothing of tenants 1 and 2
    inp2 = dict(inp)
    tg = inp["targets"].copy()
    s0 = [s for r in w.requests if r.tenant == 0 for s in r.samples]
    for s in s0:
        tg[s.target_off:s.target_off + 6] += 0.5
    inp2["targets"] = tg
    pert = M.grouped_step(w, wt, hd, inp2)
    assert pert[0]["loss"] != full[0]["loss"]
    for t in (1, 2):
        assert pert[t]["loss"] == full[t]["loss"]
        for k in full[t]["grads"]:
            np.testing.assert_array_equal(pert[t]["grads"][k], full[t]["grads"][k])


def test_block_geglu_single_token():
    lw = _layer()
    bb = _tiny_bb(glu=1)
    x = RNG.standard_normal((1, 16))
    n1 = x / np.sqrt(np.mean(x * x) + 1e-6) * lw["attn_norm"]
    vrow = lw["wv"] @ n1[0]
    h = x[0] + lw["wo"] @ np.concatenate([vrow, vrow])
    n2 = h / np.sqrt(np.mean(h * h) + 1e-6) * lw["ffn_norm"]
    g, u = lw["wg"] @ n2, lw["wu"] @ n2
    gelu = np.array([0.5 * v * (1 + math.erf(v / math.sqrt(2))) for v in g])
    ref = h + lw["wd"] @ (gelu * u)
    # tanh GELU differs from the erf form by < 1e-3 per element
    assert np.max(np.abs(M.block(bb, lw, x, 0)[0] - ref)) < 1e-3 * np.abs(lw["wd"]).sum(axis=1).max()


def test_block_zero_query_weights_average_unrotated_values():
    # W_q = 0 makes every query zero, so attention is uniform over the sample
    # and returns the plain mean of the (unrotated) value rows.
    lw = _layer()
    lw["wq"][:] = 0
    lw["wd"][:] = 0
    bb = _tiny_bb()
    x = RNG.standard_normal((5, 16))
    n1 = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + 1e-6) * lw["attn_norm"]
    vmean = (n1 @ lw["wv"].T).mean(axis=0)
    ref = x + (lw["wo"] @ np.concatenate([vmean, vmean]))[None, :]
    np.testing.assert_allclose(M.block(bb, lw, x, 0), ref, rtol=1e-12)
