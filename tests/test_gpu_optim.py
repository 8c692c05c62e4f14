"""Tenant-private head optimizer step (AdamW) and gradient accumulation
through the C ABI, against the AdamW oracle; only the group's tenants move."""
import numpy as np
import pytest
import torch

import synth
from oracle import optim as O
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.gpu_helpers import f64
from tests.helpers import oracle_requests, rel_err

pytestmark = pytest.mark.gpu

HP = dict(lr=1e-2, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)
# the C ABI carries the hyperparameters as fp32: the oracle gets the same values
HP32 = {k: float(np.float32(v)) for k, v in HP.items()}


def _close(got, ref, rtol, atol=0.0):
    # element-wise: |got - ref| <= rtol |ref| + atol (fp32 arithmetic vs fp64)
    err = np.abs(got - ref) - (rtol * np.abs(ref) + atol)
    return float(err.max()) <= 0.0


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _query_head_setup(tenants):
    """Three query-head tenants of the 2B-class workload on seeded random
    hidden rows (no backbone needed), forward and backward done."""
    w = synth.make_workload("mqa2b").subset([0, 1, 2])
    hw = synth.make_head_weights(w)
    inp = synth.make_inputs(w)
    heads = R.DeviceHeads(w.tenants, w.backbone.d,
                          [{k: v.cuda() for k, v in h.items()} for h in hw])
    ws_sub = w.subset(tenants)
    plan = J.jnx_group_plan(ws_sub.schemas(), oracle_requests(ws_sub), len(w.tenants), 1 << 30,
                            1 << 30)
    g = R.DeviceGroup(plan)
    X = (torch.randn((plan.n_tokens, w.backbone.d), generator=torch.Generator().manual_seed(5))
         .to(torch.bfloat16).cuda())
    ws = torch.zeros(heads.workspace_bytes(g), dtype=torch.uint8, device="cuda")
    tg = inp["targets"].cuda()
    preds = torch.zeros_like(tg)
    loss = torch.zeros((len(w.tenants),), device="cuda")
    heads.forward(g, None, X, tg, preds, loss, ws)
    return w, heads, g, X, tg, ws


def _mlp_setup():
    w = synth.make_workload("tiny")
    hw = synth.make_head_weights(w)
    inp = synth.make_inputs(w)
    heads = R.DeviceHeads(w.tenants, w.backbone.d,
                          [{k: v.cuda() for k, v in h.items()} for h in hw])
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    pooled = torch.randn((plan.n_samples, w.backbone.d),
                         generator=torch.Generator().manual_seed(9)).cuda()
    ws = torch.zeros(heads.workspace_bytes(g), dtype=torch.uint8, device="cuda")
    tg = inp["targets"].cuda()
    preds = torch.zeros_like(tg)
    loss = torch.zeros((len(w.tenants),), device="cuda")
    heads.forward(g, pooled, None, tg, preds, loss, ws)
    return w, heads, g, pooled, tg, ws


def _check_adamw(heads, tenants_in, tenants_all, steps=3):
    heads.init_optimizer()
    before = {t: {k: {q: a.clone() for q, a in d.items()} for k, d in heads.opt_state[t].items()}
              for t in tenants_all}
    params0 = {t: {k: heads.keep[t][k].clone() for k in heads.opt_state[t]} for t in tenants_all}
    ref = {t: {k: (f64(d["master"]), np.zeros(d["master"].shape), np.zeros(d["master"].shape))
               for k, d in before[t].items()} for t in tenants_in}
    for step in range(1, steps + 1):
        heads.adamw_step(heads._group, **HP)
        torch.cuda.synchronize()
        for t in tenants_in:
            assert heads.version(t) == step and heads.opt[t].step == step
            for k, d in heads.opt_state[t].items():
                p, m, v = ref[t][k]
                p, m, v = O.adamw_step(p, f64(heads.grads[t][k]), m, v, step, **HP32)
                ref[t][k] = (p, m, v)
                # a handful of fp32 roundings per value.  The master's error
                # scale is the update lr * (mhat / (sqrt(vhat) + eps) + wd p),
                # |.| <~ 3e-2: a few fp32 ulps of it over three steps stay
                # below 1e-7 (a wrong sign or bias correction is off by ~1e-2)
                assert _close(f64(d["m"]), m, 4e-6), (t, k, step)
                assert _close(f64(d["v"]), v, 4e-6), (t, k, step)
                assert _close(f64(d["master"]), p, 1e-6, 1e-7), (t, k, step)
                # the bf16 parameter the forward reads is the rounded master
                assert torch.equal(heads.keep[t][k], d["master"].to(torch.bfloat16)), (t, k)
    for t in set(tenants_all) - set(tenants_in):
        assert heads.version(t) == 0 and heads.opt[t].step == 0
        for k, d in heads.opt_state[t].items():
            assert torch.equal(heads.keep[t][k], params0[t][k])
            for q in ("master", "m", "v"):
                assert torch.equal(d[q], before[t][k][q])


def test_adamw_mlp_heads_vs_oracle():
    w, heads, g, pooled, tg, ws = _mlp_setup()
    heads.backward(g, pooled, None, tg, ws)
    heads._group = g
    _check_adamw(heads, [0, 1], [0, 1])


def test_adamw_query_heads_only_the_group_moves():
    w, heads, g, X, tg, ws = _query_head_setup([0, 2])
    heads.backward(g, None, X, tg, ws)
    heads._group = g
    _check_adamw(heads, [0, 2], [0, 1, 2])


@pytest.mark.parametrize("kind", ["mlp", "xattn"])
def test_gradient_accumulation_adds(kind):
    if kind == "mlp":
        w, heads, g, feat, tg, ws = _mlp_setup()
        args = (feat, None)
    else:
        w, heads, g, feat, tg, ws = _query_head_setup([0, 1, 2])
        args = (None, feat)
    heads.backward(g, *args, tg, ws)
    one = [{k: v.clone() for k, v in gr.items()} for gr in heads.grads]
    heads.backward(g, *args, tg, ws, accumulate=True)
    torch.cuda.synchronize()
    for t in g.plan.slot_tenant.tolist():
        for k, v in heads.grads[t].items():
            assert torch.equal(v, 2 * one[t][k]), (t, k)
    # overwrite mode goes back to one backward's gradients
    heads.backward(g, *args, tg, ws)
    torch.cuda.synchronize()
    for t in g.plan.slot_tenant.tolist():
        for k, v in heads.grads[t].items():
            assert torch.equal(v, one[t][k]), (t, k)


def test_adamw_rejects_bad_hyperparameters():
    w, heads, g, pooled, tg, ws = _mlp_setup()
    heads.init_optimizer()
    for bad in (dict(lr=-1.0), dict(beta1=1.0), dict(beta2=-0.1), dict(weight_decay=-1.0)):
        with pytest.raises(J.JnxError):
            heads.adamw_step(g, **dict(HP, **bad))
    assert heads.version(0) == 0


def test_tenant_adamw_on_stacked_slices_only_the_named_tenants_move():
    # the generic entry point (jnx_adamw_tensors) on stacked per-tenant
    # tensors, as the LoRA adapters and flow experts hold them
    g = torch.Generator().manual_seed(12)
    params = [torch.randn(3, 40, 24, generator=g).to(torch.bfloat16).cuda(),
              torch.randn(3, 7, generator=g).to(torch.bfloat16).cuda()]
    grads = [torch.randn(p.shape, generator=g).cuda() for p in params]
    p0 = [p.clone() for p in params]
    opt = R.TenantAdamW(list(zip(params, grads)))
    ref = {(i, t): (f64(params[i][t]), np.zeros(params[i][t].shape), np.zeros(params[i][t].shape))
           for i in range(2) for t in (0, 2)}
    for step in (1, 2, 3):
        opt.step([0, 2], **HP)
        torch.cuda.synchronize()
        for (i, t), (p, m, v) in ref.items():
            p, m, v = O.adamw_step(p, f64(grads[i][t]), m, v, step, **HP32)
            ref[(i, t)] = (p, m, v)
            assert opt.steps(i, t) == step
            assert _close(f64(opt.m[i][t]), m, 4e-6)
            assert _close(f64(opt.v[i][t]), v, 4e-6)
            assert _close(f64(opt.master[i][t]), p, 1e-6, 1e-7)
            assert torch.equal(params[i][t], opt.master[i][t].to(torch.bfloat16))
    for i in range(2):
        assert torch.equal(params[i][1], p0[i][1])  # tenant 1 not named: untouched
        assert opt.steps(i, 1) == 0


def test_flow_expert_and_adapter_parameter_pairs():
    # the accessors pair every trainable tensor with a gradient of its shape
    w = synth.make_workload("zipf2b", n_layers=1)
    bw = synth.make_backbone_weights(w.subset([0]), device="cuda")
    bb = R.DeviceBackbone(w.backbone, bw, n_tenants=len(w.tenants))
    bb.prepare_backward()
    pairs = bb.lora_pairs()
    assert len(pairs) == 8
    for p, gr in pairs:
        assert p.shape == gr.shape and p.dtype == torch.bfloat16 and gr.dtype == torch.float32
    dims = dict(n_tenants=2, d_model=256, d_ff=256, chunk=4, action_dim=3, d_in=256)
    fw = synth.make_flow_weights(2, 256, 256, 2, 4, 3, 256, 5, device="cuda")
    fh = R.DeviceFlowHeads(dims, fw)
    fp = fh.param_pairs()
    assert len(fp) == 9 + 2 * 5
    for p, gr in fp:
        assert p.shape == gr.shape
