"""Pins of the LoRA-backward oracle (oracle/backward.py): closed-form
identities of its pieces and central finite differences of the forward
oracle's loss, so that a dropped term, a wrong sign or a transposed operand
in any step of the chain rule fails one of them."""
import math

import numpy as np
import pytest

import synth
from oracle import backward as B
from oracle import model as M

RNG = np.random.default_rng(11)


def _fd(fn, arr, idx, h=1e-6):
    flat = arr.reshape(-1)
    old = flat[idx]
    flat[idx] = old + h
    lp = fn()
    flat[idx] = old - h
    lm = fn()
    flat[idx] = old
    return (lp - lm) / (2 * h)


def _check(fd, an, scale, rtol=1e-6):
    assert abs(fd - an) <= rtol * max(abs(fd), scale) + 1e-10, (fd, an, scale)


# ---------------- pieces ------------------------------------------------------

def test_rope_backward_is_the_adjoint_and_the_inverse():
    x = RNG.standard_normal((9, 3, 16))
    y = RNG.standard_normal((9, 3, 16))
    pos = np.arange(9) * 7
    fx = M.rope(x, pos, 1e4)
    np.testing.assert_allclose(np.sum(fx * y), np.sum(x * B.rope_backward(y, pos, 1e4)),
                               rtol=1e-13)
    # a rotation's transpose is its inverse
    np.testing.assert_allclose(B.rope_backward(fx, pos, 1e4), x, rtol=1e-12, atol=1e-13)


def test_rmsnorm_backward_finite_differences():
    x = RNG.standard_normal((4, 24))
    g = 1 + 0.3 * RNG.standard_normal(24)
    dn = RNG.standard_normal((4, 24))
    an = B.rmsnorm_backward(x, g, 1e-6, dn)
    fn = lambda: float(np.sum(dn * M.rmsnorm(x, g, 1e-6)))
    for idx in RNG.choice(x.size, 20, replace=False):
        _check(_fd(fn, x, idx), an.reshape(-1)[idx], np.abs(an).max())
    # with eps = 0 a row scaled by c > 0 has the same normed output, so the
    # derivative along x itself vanishes: dx . x = 0 per row
    an0 = B.rmsnorm_backward(x, g, 0.0, dn)
    np.testing.assert_allclose(np.sum(an0 * x, axis=1), 0.0, atol=1e-12)
    assert np.abs(np.sum(an * x, axis=1)).max() > 1e-9  # eps > 0 breaks it


def test_gelu_tanh_grad_finite_differences_and_values():
    z = np.linspace(-4, 4, 33)
    fd = (M.gelu_tanh(z + 1e-6) - M.gelu_tanh(z - 1e-6)) / 2e-6
    np.testing.assert_allclose(B.gelu_tanh_grad(z), fd, rtol=1e-7, atol=1e-9)
    assert B.gelu_tanh_grad(np.array([0.0]))[0] == 0.5


def test_attention_backward_finite_differences_with_kv_groups():
    L, H, Hkv, hd = 6, 4, 2, 8
    q = RNG.standard_normal((L, H, hd))
    k = RNG.standard_normal((L, Hkv, hd))
    v = RNG.standard_normal((L, Hkv, hd))
    do = RNG.standard_normal((L, H, hd))
    dq, dk, dv = B.attention_backward(q, k, v, do)
    fn = lambda: float(np.sum(do * M.attention(q, k, v)))
    for arr, an in ((q, dq), (k, dk), (v, dv)):
        for idx in RNG.choice(arr.size, 16, replace=False):
            _check(_fd(fn, arr, idx), an.reshape(-1)[idx], np.abs(an).max())


def test_attention_backward_single_key():
    # one key: P = 1 whatever q, so dq = 0 and dk = 0, and dv sums do over
    # the query heads that share the K/V head
    q = RNG.standard_normal((1, 4, 8))
    k = RNG.standard_normal((1, 2, 8))
    v = RNG.standard_normal((1, 2, 8))
    do = RNG.standard_normal((1, 4, 8))
    dq, dk, dv = B.attention_backward(q, k, v, do)
    assert np.all(np.abs(dq) < 1e-15) and np.all(np.abs(dk) < 1e-15)
    np.testing.assert_allclose(dv[0, 0], do[0, 0] + do[0, 1], rtol=1e-14)
    np.testing.assert_allclose(dv[0, 1], do[0, 2] + do[0, 3], rtol=1e-14)


def _bb(glu):
    return dict(n_heads=4, n_kv_heads=2, head_dim=8, eps=1e-6, rope_theta=1e4, glu=glu,
                vision_tokens=2, d=16)


def _layer(d=16, H=4, Hkv=2, hd=8, F=24, r=3, T=2, scale=0.3):
    lw = dict(attn_norm=1 + 0.1 * RNG.standard_normal(d),
              wq=scale * RNG.standard_normal((H * hd, d)),
              wk=scale * RNG.standard_normal((Hkv * hd, d)),
              wv=scale * RNG.standard_normal((Hkv * hd, d)),
              wo=scale * RNG.standard_normal((d, H * hd)),
              ffn_norm=1 + 0.1 * RNG.standard_normal(d),
              wg=scale * RNG.standard_normal((F, d)), wu=scale * RNG.standard_normal((F, d)),
              wd=scale * RNG.standard_normal((d, F)))
    for nm, din, dout in (("q", d, H * hd), ("k", d, Hkv * hd), ("v", d, Hkv * hd),
                          ("o", H * hd, d)):
        lw["lora_a_" + nm] = scale * RNG.standard_normal((T, r, din))
        lw["lora_b_" + nm] = scale * RNG.standard_normal((T, dout, r))
    return lw


@pytest.mark.parametrize("glu", [0, 1])
def test_block_backward_finite_differences(glu):
    bb, lw = _bb(glu), _layer()
    x = RNG.standard_normal((5, 16))
    dy = RNG.standard_normal((5, 16))
    out, c = B.block_forward(bb, lw, x, 1)
    np.testing.assert_allclose(out, M.block(bb, lw, x, 1), rtol=1e-13)  # same forward
    dx, g = B.block_backward(bb, lw, c, dy, 1)
    fn = lambda: float(np.sum(dy * M.block(bb, lw, x, 1)))
    for idx in RNG.choice(x.size, 12, replace=False):
        _check(_fd(fn, x, idx), dx.reshape(-1)[idx], np.abs(dx).max())
    for nm in ("q", "k", "v", "o"):
        for kind in ("a", "b"):
            an = g[kind + "_" + nm]
            arr = lw["lora_%s_%s" % (kind, nm)][1]
            assert an.shape == arr.shape
            for idx in RNG.choice(arr.size, 6, replace=False):
                _check(_fd(fn, arr, idx), an.reshape(-1)[idx], np.abs(an).max())
    # the other tenant's adapter does not enter this sample
    fd0 = _fd(fn, lw["lora_a_q"][0], 0)
    assert fd0 == 0.0


def test_adapter_gradients_with_zero_b():
    # B = 0: the adapter adds nothing and dA = (gY B)^T x vanishes exactly
    bb, lw = _bb(0), _layer()
    for nm in ("q", "k", "v", "o"):
        lw["lora_b_" + nm][:] = 0.0
    x = RNG.standard_normal((4, 16))
    _, c = B.block_forward(bb, lw, x, 0)
    _, g = B.block_backward(bb, lw, c, RNG.standard_normal((4, 16)), 0)
    for nm in ("q", "k", "v", "o"):
        assert np.all(g["a_" + nm] == 0.0)
        assert np.abs(g["b_" + nm]).max() > 0.0


# ---------------- heads ---------------------------------------------------------

def test_head_feature_grads_finite_differences():
    d = 12
    mlp = dict(w1=0.3 * RNG.standard_normal((10, d)), b1=0.1 * RNG.standard_normal(10),
               w2=0.3 * RNG.standard_normal((6, 10)), b2=0.1 * RNG.standard_normal(6))
    xat = dict(q=RNG.standard_normal((3, 4)), wk=0.5 * RNG.standard_normal((4, d)),
               wv=0.5 * RNG.standard_normal((4, d)), wout=0.3 * RNG.standard_normal((5, 12)),
               bout=0.1 * RNG.standard_normal(5))
    for kind, hw, feats, T in (
            (0, mlp, [RNG.standard_normal(d) for _ in range(3)], RNG.uniform(-1, 1, (3, 6))),
            (1, xat, [RNG.standard_normal((L, d)) for L in (1, 4, 6)],
             RNG.uniform(-1, 1, (3, 5)))):
        an = B.head_feature_grads(kind, hw, feats, T)
        fn = lambda: M.tenant_step(kind, hw, feats, T)[0]
        for f, a in zip(feats, an):
            for idx in RNG.choice(f.size, min(f.size, 8), replace=False):
                _check(_fd(fn, f, idx), a.reshape(-1)[idx], np.abs(a).max())


# ---------------- the whole path ---------------------------------------------------

def _lora_workload(glu):
    bb = synth.Backbone(n_layers=2, d=32, n_heads=4, n_kv_heads=2, head_dim=8, d_ff=40,
                        vision_tokens=3, vocab=50, qk_std=0.3, glu=glu, lora_rank=4)
    tenants = [synth.Tenant(synth.HEAD_MLP, chunk=2, action_dim=3, d_hidden=12, max_images=2),
               synth.Tenant(synth.HEAD_XATTN, chunk=2, action_dim=2, n_queries=3, q_dim=8,
                            max_images=2)]
    per = [[synth.Sample(1, 2), synth.Sample(0, 4)], [synth.Sample(2, 1), synth.Sample(1, 0)]]
    w = synth.custom_workload(bb, tenants, per, req_batch=1, seed=21)
    wt = M.widen_tree(synth.to_numpy_tree(synth.make_backbone_weights(w, std=0.25)))
    hd = M.widen_tree(synth.to_numpy_tree(synth.make_head_weights(w, std=0.3)))
    inp = synth.to_numpy_tree(synth.make_inputs(w))
    return w, wt, hd, inp


@pytest.mark.parametrize("glu", [0, 1])
def test_lora_step_finite_differences_of_the_forward_oracle(glu):
    w, wt, hw, inp = _lora_workload(glu)
    res = B.lora_step(w, wt, hw, inp)
    fwd = M.grouped_step(w, wt, hw, inp)
    for t in (0, 1):
        assert res[t]["loss"] == pytest.approx(fwd[t]["loss"], rel=1e-13)
        np.testing.assert_allclose(res[t]["pred"], fwd[t]["pred"], rtol=1e-13)
        fn = lambda: M.grouped_step(w, wt, hw, inp, tenants=[t])[t]["loss"]
        for l in range(2):
            for key, an in res[t]["lora"][l].items():
                kind, nm = key.split("_")
                arr = wt["layers"][l]["lora_%s_%s" % (kind, nm)][t]
                for idx in RNG.choice(arr.size, 4, replace=False):
                    _check(_fd(fn, arr, idx), an.reshape(-1)[idx], np.abs(an).max(), 1e-5)
        # a random direction through every adapter of the tenant at once
        dirs = {}
        for l in range(2):
            for nm in B.PARTS:
                for kind in ("a", "b"):
                    dirs[(l, kind, nm)] = RNG.standard_normal(
                        wt["layers"][l]["lora_%s_%s" % (kind, nm)][t].shape)

        def shifted(eps):
            for (l, kind, nm), v in dirs.items():
                wt["layers"][l]["lora_%s_%s" % (kind, nm)][t] += eps * v
            out = fn()
            for (l, kind, nm), v in dirs.items():
                wt["layers"][l]["lora_%s_%s" % (kind, nm)][t] -= eps * v
            return out

        h = 1e-6
        fd = (shifted(h) - shifted(-h)) / (2 * h)
        an = sum(float(np.sum(res[t]["lora"][l][kind + "_" + nm] * v))
                 for (l, kind, nm), v in dirs.items())
        assert fd == pytest.approx(an, rel=1e-6, abs=1e-9)


def test_lora_step_other_tenants_adapters_do_not_matter():
    w, wt, hw, inp = _lora_workload(0)
    ref = B.lora_step(w, wt, hw, inp, tenants=[0])[0]
    for L in wt["layers"]:
        for nm in B.PARTS:
            L["lora_a_" + nm][1] += 1.0
            L["lora_b_" + nm][1] *= -2.0
    got = B.lora_step(w, wt, hw, inp, tenants=[0])[0]
    assert got["loss"] == ref["loss"]
    for a, b in zip(got["lora"], ref["lora"]):
        for k in a:
            np.testing.assert_array_equal(a[k], b[k])


def test_d_hidden_is_the_feature_gradient_spread_over_rows():
    # MLP tenant: every row of a sample carries dfeature / L
    w, wt, hw, inp = _lora_workload(0)
    res = B.lora_step(w, wt, hw, inp, tenants=[0])[0]
    for dh in res["d_hidden"]:
        np.testing.assert_allclose(dh, np.tile(dh[0], (dh.shape[0], 1)), rtol=1e-15)
    assert math.isfinite(res["loss"])
