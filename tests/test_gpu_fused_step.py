"""The heads backward with the tenant-private AdamW step fused into it
(jnx_heads_backward_adamw), through the C ABI.  Its result is defined as the
separate backward (jnx_heads_backward / _accumulate) followed by the
separate optimizer step (jnx_heads_adamw), which tests/test_gpu_optim.py
checks against the AdamW oracle.  So the fused path is held to that result
bit for bit over two training steps: every bf16 parameter, fp32 master and
moment, the per-tenant step and policy-version counters, the feature
gradient, with and without gradient accumulation, for MLP heads at the
7B-class shapes and for query heads; tenants outside the group are not
touched (App. A: only the microbatch's tenant's optimizer steps)."""
import pytest
import torch

import synth
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.helpers import oracle_requests

pytestmark = pytest.mark.gpu

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _pair(w, hw):
    """Two head sets with the same initial parameters and optimizer state."""
    out = []
    for _ in range(2):
        h = R.DeviceHeads(w.tenants, w.backbone.d,
                          [{k: v.clone().cuda() for k, v in x.items()} for x in hw])
        h.init_optimizer()
        out.append(h)
    return out


def _state(h):
    ts = []
    for t in range(h.n):
        for k in sorted(h.keep[t]):
            ts.append((t, k, "param", h.keep[t][k]))
            st = h.opt_state[t][k]
            ts += [(t, k, c, st[c]) for c in ("master", "m", "v")]
    return ts


def _assert_same(a, b, step):
    bad = []
    for (t, k, c, x), (_, _, _, y) in zip(_state(a), _state(b)):
        if not torch.equal(x, y):
            d = (x.float() - y.float()).abs()
            bad.append(f"tenant {t} {k} {c}: {int((d > 0).sum())} of {d.numel()} differ, "
                       f"max {float(d.max()):.3e} (|ref| max {float(x.float().abs().max()):.3e})")
    assert not bad, (step, bad[:8])
    for t in range(a.n):
        assert a.version(t) == b.version(t) and a.opt[t].step == b.opt[t].step


def _run(w, tenants, feat_fn, accumulate, with_dh):
    hw = synth.make_head_weights(w)
    inp = synth.make_inputs(w)
    sep, fused = _pair(w, hw)
    wsub = w.subset(tenants)
    plan = J.jnx_group_plan(wsub.schemas(), oracle_requests(wsub), len(w.tenants), 1 << 30,
                            1 << 30)
    g = R.DeviceGroup(plan)
    pooled, hidden = feat_fn(plan)
    tg = inp["targets"].cuda()
    ws = [torch.zeros(h.workspace_bytes(g), dtype=torch.uint8, device="cuda")
          for h in (sep, fused)]
    untouched = {t: [x.clone() for x in _state_of(fused, t)] for t in range(len(w.tenants))
                 if t not in tenants}
    d = w.backbone.d
    for step in range(2):
        dh = [torch.full((plan.n_tokens, d), float("nan"), device="cuda") for _ in range(2)]
        outs = []
        for i, h in enumerate((sep, fused)):
            preds = torch.zeros_like(tg)
            loss = torch.zeros((len(w.tenants),), device="cuda")
            h.forward(g, pooled, hidden, tg, preds, loss, ws[i])
            outs.append((preds, loss))
            if accumulate:  # an earlier microbatch's gradients, then this one's
                h.backward(g, pooled, hidden, tg, ws[i])
        # equal parameters give equal forwards
        assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1]), step
        if with_dh:
            sep.backward_input(g, pooled, hidden, tg, dh[0], ws[0])
            if accumulate:  # backward_input overwrote: add the earlier microbatch again
                sep.backward(g, pooled, hidden, tg, ws[0], accumulate=True)
        else:
            sep.backward(g, pooled, hidden, tg, ws[0], accumulate=accumulate)
        sep.adamw_step(g, **HP)
        fused.backward_adamw(g, pooled, hidden, tg, ws[1], accumulate=accumulate,
                             d_hidden=dh[1] if with_dh else None, **HP)
        torch.cuda.synchronize()
        R.check_status(ws[0])
        R.check_status(ws[1])
        _assert_same(sep, fused, step)
        if with_dh:
            assert torch.equal(dh[0], dh[1]), step
    for t in tenants:
        assert fused.version(t) == 2
    for t, before in untouched.items():
        assert fused.version(t) == 0
        for x, y in zip(before, _state_of(fused, t)):
            assert torch.equal(x, y), t


def _state_of(h, t):
    ts = []
    for k in sorted(h.keep[t]):
        st = h.opt_state[t][k]
        ts += [h.keep[t][k], st["master"], st["m"], st["v"]]
    return ts


@pytest.mark.parametrize("accumulate,with_dh", [(False, False), (True, False), (False, True)])
def test_fused_step_equals_backward_then_adamw_mlp_7b_heads(accumulate, with_dh):
    """32 MLP heads of the 7B-class group (4096 -> 1024 -> 56), 4 of them in
    the group, on seeded random pooled features."""
    w = synth.make_workload("llama7b")

    def feats(plan):
        p = torch.randn((plan.n_samples, w.backbone.d), generator=torch.Generator().manual_seed(3))
        return p.cuda(), None

    _run(w, [0, 5, 30, 31], feats, accumulate, with_dh)


@pytest.mark.parametrize("accumulate,with_dh", [(False, False), (True, False), (False, True)])
def test_fused_step_equals_backward_then_adamw_query_heads(accumulate, with_dh):
    """Query heads (32 queries x 256, d = 2048) of the 2B-class workload,
    two of three tenants in the group, on seeded random hidden rows."""
    w = synth.make_workload("mqa2b").subset([0, 1, 2])

    def feats(plan):
        X = torch.randn((plan.n_tokens, w.backbone.d), generator=torch.Generator().manual_seed(5))
        return None, X.to(torch.bfloat16).cuda()

    _run(w, [0, 2], feats, accumulate, with_dh)


def test_fused_step_refuses_missing_optimizer_state():
    w = synth.make_workload("tiny")
    hw = synth.make_head_weights(w)
    h = R.DeviceHeads(w.tenants, w.backbone.d, [{k: v.cuda() for k, v in x.items()} for x in hw])
    h.init_optimizer()
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    ws = torch.zeros(h.workspace_bytes(g), dtype=torch.uint8, device="cuda")
    pooled = torch.zeros((plan.n_samples, w.backbone.d), device="cuda")
    tg = synth.make_inputs(w)["targets"].cuda()
    h.opt[1].m[0] = None
    before = [x.clone() for x in _state_of(h, 0)]
    with pytest.raises(J.JnxError, match="null state"):
        h.backward_adamw(g, pooled, None, tg, ws, **HP)
    torch.cuda.synchronize()
    for x, y in zip(before, _state_of(h, 0)):
        assert torch.equal(x, y)
    assert h.version(0) == 0


@pytest.mark.parametrize("name", ["llama7b", "mqa2b"])
def test_heads_forward_and_backward_are_deterministic(name):
    """The same inputs give the same bits on every run (no atomics, fixed
    reduction orders), in two workspaces of their own."""
    w = synth.make_workload(name)
    w = w.subset([0, 1, 2]) if name == "mqa2b" else w.subset([0, 5, 30, 31])
    hw = synth.make_head_weights(w)
    h = R.DeviceHeads(w.tenants, w.backbone.d, [{k: v.cuda() for k, v in x.items()} for x in hw])
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    gen = torch.Generator().manual_seed(9)
    if name == "mqa2b":
        pooled, hidden = None, torch.randn((plan.n_tokens, w.backbone.d), generator=gen).to(
            torch.bfloat16).cuda()
    else:
        pooled, hidden = torch.randn((plan.n_samples, w.backbone.d), generator=gen).cuda(), None
    tg = synth.make_inputs(w)["targets"].cuda()
    runs = []
    for r in range(6):
        ws = torch.zeros(h.workspace_bytes(g), dtype=torch.uint8, device="cuda")
        preds = torch.zeros_like(tg)
        loss = torch.zeros((len(w.tenants),), device="cuda")
        h.forward(g, pooled, hidden, tg, preds, loss, ws)
        h.backward(g, pooled, hidden, tg, ws)
        torch.cuda.synchronize()
        runs.append([preds.clone(), loss.clone()] +
                    [v.clone() for gr in h.grads for v in gr.values()])
    for r in range(1, len(runs)):
        for i, (a, b) in enumerate(zip(runs[0], runs[r])):
            assert torch.equal(a, b), (r, i, int((a != b).sum()))
