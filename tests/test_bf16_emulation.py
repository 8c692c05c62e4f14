"""Pins of the test-side bf16 rounding-point emulation (tests/bf16_emulation.py).

The emulation sets the floor that the full-depth GPU parity tests compare
against, so it is pinned to things other than itself: its rounding helper to
PyTorch's own fp32 -> bf16 conversion and hand-worked ties; with every
rounding switched off it must reproduce the oracle's forward to 1e-12 of rms
(both forms of the RMSNorm it can model, with adapters, grouped K/V heads
and GeGLU); and each rounding point must act on its own, by the amount its
format implies."""
import numpy as np
import pytest
import torch

import synth
from oracle import model as M
from tests import bf16_emulation as E
from tests.helpers import rel_err


def test_bf16_rounding_hand_ties_and_torch():
    # bf16 keeps 7 mantissa bits: 1 + 2^-8 is a tie that goes to the even 1.0;
    # 1 + 3 2^-8 is a tie that goes to the even 1 + 2^-6
    assert E.bf16(np.array([1 + 2 ** -8]))[0] == 1.0
    assert E.bf16(np.array([1 + 3 * 2 ** -8]))[0] == 1 + 2 ** -6
    assert E.bf16(np.array([-(1 + 3 * 2 ** -8)]))[0] == -(1 + 2 ** -6)
    assert E.bf16(np.array([1 + 2 ** -8 + 2 ** -20]))[0] == 1 + 2 ** -7
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-30, 30, 20000),
                        [0.0, -0.0, 65504.0, 3.0e38, 1e-40]])
    want = torch.tensor(x, dtype=torch.float64).to(torch.float32).to(torch.bfloat16)
    np.testing.assert_array_equal(E.bf16(x), want.to(torch.float64).numpy())


def _workload(lora=True, glu=synth.GLU_GEGLU):
    bb = synth.Backbone(n_layers=2, d=64, n_heads=4, n_kv_heads=2, head_dim=16, d_ff=96,
                        glu=glu, lora_rank=4 if lora else 0, vision_tokens=4, vocab=50,
                        qk_std=0.2)
    tenants = [synth.Tenant(synth.HEAD_MLP, chunk=2, action_dim=3, d_hidden=16, max_images=2)
               for _ in range(3)]
    per = [[synth.Sample(1, 3), synth.Sample(2, 5)], [synth.Sample(2, 1)],
           [synth.Sample(1, 6), synth.Sample(0, 2)]]
    return synth.custom_workload(bb, tenants, per, req_batch=1, seed=11)


def _inputs(w):
    # weights of std 0.1 (gain about 0.8 per projection at d = 64) keep the
    # two blocks from amplifying a rounding far beyond its own size
    wt = synth.to_numpy_tree(synth.make_backbone_weights(w, std=0.1))
    inp = synth.to_numpy_tree(synth.make_inputs(w))
    bb = M.backbone_dict(w)
    samples = [(r.tenant, s) for r in w.requests for s in r.samples]
    xs = [M.sample_embeddings(bb, vars(s), inp["vision"], inp["text_ids"], wt["text_table"])
          for _, s in samples]
    return wt, bb, xs, [t for t, _ in samples]


@pytest.mark.parametrize("lora,glu", [(True, synth.GLU_GEGLU), (False, synth.GLU_SWIGLU)])
@pytest.mark.parametrize("folds", [(False, False), (True, True), (True, False)])
def test_without_rounding_the_emulation_is_the_oracle(lora, glu, folds):
    w = _workload(lora, glu)
    wt, bb, xs, tenants = _inputs(w)
    rows = E.forward(w.backbone, wt, xs, tenants, rounding=E.NONE, pool=False, folds=folds)
    pooled = E.forward(w.backbone, wt, xs, tenants, rounding=E.NONE, folds=folds)
    for x, t, r, p in zip(xs, tenants, rows, pooled):
        ref = M.backbone_sample(bb, wt, x, t)
        assert rel_err(r, ref) < 1e-12
        assert rel_err(p, M.mean_pool(ref)) < 1e-12


def _floor(w, rounding, pool=True, folds=None):
    wt, bb, xs, tenants = _inputs(w)
    got = E.forward(w.backbone, wt, xs, tenants, rounding=rounding, pool=pool, folds=folds)
    errs = []
    for x, t, g in zip(xs, tenants, got):
        ref = M.backbone_sample(bb, wt, x, t)
        errs.append(rel_err(g, M.mean_pool(ref) if pool else ref))
    return max(errs)


@pytest.mark.parametrize("point", [p for p in E.ALL if p not in ("resid", "hidden", "ds")])
def test_each_bf16_point_acts_alone_at_bf16_size(point):
    # one bf16 rounding point alone moves the result by about 2^-9 of the
    # values it touches, carried through at most two blocks: above 1e-5 and
    # below 3e-2 of rms
    e = _floor(_workload(), (point,), pool=False, folds=(True, True))
    assert 1e-5 < e < 3e-2, (point, e)


def test_fp32_residual_and_bf16_hidden_rounding_sizes():
    w = _workload()
    e = _floor(w, ("resid",), pool=False)
    assert 1e-10 < e < 1e-6, e               # fp32: about 2^-24 per update
    # one bf16 rounding of the rows themselves: at most 2^-8 of an element,
    # whose peak is a few times rms
    e = _floor(w, ("hidden",), pool=False)
    assert 2 ** -10 < e < 2 ** -5, e
    assert _floor(w, ("hidden",), pool=True) < 1e-12  # pooled features are not stored rows


def test_adapter_rounding_needs_adapters_and_fold_changes_the_operand():
    w = _workload(lora=False)
    assert _floor(w, ("lora_t",), pool=False) < 1e-12
    # the folded and unfolded norm operands round different values
    a = _floor(_workload(), ("norm",), pool=False, folds=(True, True))
    b = _floor(_workload(), ("norm",), pool=False, folds=(False, False))
    assert a != b and max(a, b) < 3e-2


def test_unknown_rounding_point_is_refused():
    with pytest.raises(ValueError):
        E.Emulation(_workload().backbone, [], [], rounding=("nrom",))


def _qkv(L=37, H=4, Hkv=2, hd=16, seed=5, std=1.0):
    rng = np.random.default_rng(seed)
    q = E.bf16(rng.standard_normal((L, H, hd)) * std)
    k = E.bf16(rng.standard_normal((L, Hkv, hd)) * std)
    v = E.bf16(rng.standard_normal((L, Hkv, hd)))
    do = E.bf16(rng.standard_normal((L, H, hd)))
    return q, k, v, do


def test_attention_functions_without_rounding_are_the_oracles():
    from oracle import backward as B
    q, k, v, do = _qkv()
    ref = M.attention(q, k, v).reshape(q.shape[0], -1)
    assert rel_err(E.attention(q, k, v, E.NONE), ref) < 1e-13
    for got, want in zip(E.attention_backward(q, k, v, do, E.NONE),
                         B.attention_backward(q, k, v, do)):
        assert rel_err(got, want) < 1e-12


def test_attention_rounding_points_act_at_bf16_size():
    q, k, v, do = _qkv(std=0.5)
    ref = M.attention(q, k, v).reshape(q.shape[0], -1)
    e_p = rel_err(E.attention(q, k, v, ("p",)), ref)
    e_o = rel_err(E.attention(q, k, v, ("attn_out",)), ref)
    assert 1e-5 < e_p < 2e-2 and 1e-5 < e_o < 2e-2
    want = E.attention_backward(q, k, v, do, E.NONE)
    for pt, moved in (("p", (False, False, True)), ("ds", (True, True, False)),
                      ("attn_out", (True, True, False))):
        got = E.attention_backward(q, k, v, do, (pt,))
        for g, w_, m in zip(got, want, moved):
            e = rel_err(g, w_)
            assert (1e-5 < e < 5e-2) if m else e == 0.0, (pt, e)
