"""Flow-matching action experts (DiT heads) as tenant-private modules,
through the C ABI, against the fp64 oracle (oracle/flow.py): the velocity,
each tenant's loss and every parameter gradient; Euler sampling; grouped ==
isolated (bit for bit); slot isolation and gradient accumulation."""
import numpy as np
import pytest
import torch

import synth
from oracle import flow as Fl
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.gpu_helpers import f64
from tests.helpers import BF16_TOL, oracle_requests, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


# Velocities, losses and Euler samples are held to the stated 2e-2
# (measured on GB300 at most 0.017, 2.4e-3 and 4.3e-3).  The parameter
# gradients are sums over the action rows of products of bf16-rounded
# factors, and their max|err|/rms is ill-conditioned: perturbing the fp64
# oracle's own parameters and context rows by relative noise of 2^-9 (2^-8)
# moves its gradients by up to 0.094 (0.177) of rms.  Measured on GB300,
# worst over every tenant and parameter: 0.054 - 0.156 (the training-step
# cases), 0.174 (the flow bench's launch configuration); the bound is 1.5x
# the worst (relative L2 of the same gradients: 1.2e-3 - 6.2e-3).
FLOW_GRAD_TOL = 0.26


def _err(what, got, ref, tol, worst):
    e = rel_err(got, ref)
    print(f"{what}: max|err|/rms {e:.4e}")
    worst[0] = max(worst[0], e)
    assert e < tol, (what, e, tol)


class FlowSetup:
    def __init__(self, dm=256, F=256, nb=2, C=8, D=7, d=256, per=None, seed=3, std=0.05,
                 workload=None):
        if workload is None:
            per = per or [[synth.Sample(1, 5), synth.Sample(0, 17)],
                          [synth.Sample(2, 3)],
                          [synth.Sample(0, 1), synth.Sample(1, 40), synth.Sample(0, 9)]]
            bb = synth.Backbone(n_layers=0, d=d, n_heads=4, n_kv_heads=4, head_dim=64, d_ff=1024,
                                vision_tokens=32, vocab=100)
            tenants = [synth.Tenant(synth.HEAD_MLP, chunk=C, action_dim=D, d_hidden=64,
                                    max_images=2) for _ in per]
            workload = synth.custom_workload(bb, tenants, per, req_batch=1, seed=seed)
        self.w = workload
        T = len(self.w.tenants)
        self.dims = dict(n_tenants=T, d_model=dm, d_ff=F, chunk=C, action_dim=D, d_in=d)
        self.wt = synth.make_flow_weights(T, dm, F, nb, C, D, d, seed, device="cuda", std=std)
        self.heads = R.DeviceFlowHeads(self.dims, self.wt)
        self.nh = dm // 64
        self.C, self.D = C, D

    def plan(self, tenants=None):
        w = self.w if tenants is None else self.w.subset(tenants)
        return J.jnx_group_plan(w.schemas(), oracle_requests(w), len(self.w.tenants), 1 << 30,
                                1 << 30)

    def run(self, plan, hidden, inp, accumulate=False):
        g = R.DeviceGroup(plan)
        S = plan.n_samples
        ws = torch.zeros(max(self.heads.workspace_bytes(g), 256), dtype=torch.uint8,
                         device="cuda")
        vel = torch.full((S, self.C, self.D), float("nan"), device="cuda")
        loss = torch.full((len(self.w.tenants),), float("nan"), device="cuda")
        self.heads.forward(g, hidden, inp["actions"], inp["noise"], inp["tau"], vel, loss, ws)
        self.heads.backward(g, hidden, ws, accumulate=accumulate)
        R.check_status(ws)
        torch.cuda.synchronize()
        return g, vel, loss, ws

    def oracle_params(self, t):
        W = self.wt
        p = {k: f64(W[k][t]) for k in J.FLOW_PARAMS}
        p["blocks"] = [dict(wqkv=f64(B["w_qkv"][t]), wkvc=f64(B["w_kvc"][t]), wo=f64(B["w_o"][t]),
                            wg=f64(B["wg"][t]), wu=f64(B["wu"][t]), wd=f64(B["w_d"][t]))
                       for B in W["blocks"]]
        return p

    def unpack_gu(self, g):
        """[2F, dm] in the packed order -> (gate rows, up rows)."""
        F = self.dims["d_ff"]
        blocks = g.reshape(2 * F // 128, 128, -1)
        return blocks[0::2].reshape(F, -1), blocks[1::2].reshape(F, -1)


def _inputs(plan, C, D, seed=4):
    inp = synth.make_flow_inputs(plan.n_samples, C, D, seed, device="cuda")
    return inp


def _check(s, plan, hidden, inp, vel, loss, tol, only=None):
    H = f64(hidden)
    cu, seg = plan.cu_seqlens, plan.seg_offsets
    worst = [0.0]
    for gi, t in enumerate(plan.slot_tenant.tolist()):
        if only is not None and t not in only:
            continue
        ss = range(seg[gi], seg[gi + 1])
        ctx = [H[cu[i]:cu[i + 1]] for i in ss]
        acts = f64(inp["actions"][seg[gi]:seg[gi + 1]])
        noise = f64(inp["noise"][seg[gi]:seg[gi + 1]])
        taus = f64(inp["tau"][seg[gi]:seg[gi + 1]])
        p = s.oracle_params(t)
        ref_loss, V, G = Fl.tenant_step(p, s.nh, ctx, acts, noise, taus)
        _err(f"tenant {t} velocity", f64(vel[seg[gi]:seg[gi + 1]]), V, BF16_TOL, [0.0])
        e = abs(float(loss[t]) - ref_loss) / ref_loss
        print(f"tenant {t} loss: relative {e:.4e}")
        assert e <= BF16_TOL, ("loss", t, e)
        for k in J.FLOW_PARAMS:
            _err(f"tenant {t} grad {k}", f64(s.heads.grads[k][t]), G[k], tol, worst)
        for b, GB in enumerate(G["blocks"]):
            dg = s.heads.block_grads[b]
            pairs = [("w_qkv", GB["wqkv"]), ("w_kvc", GB["wkvc"]), ("w_o", GB["wo"]),
                     ("w_d", GB["wd"])]
            for name, ref in pairs:
                _err(f"tenant {t} block {b} grad {name}", f64(dg[name][t]), ref, tol, worst)
            gg, gu = s.unpack_gu(f64(dg["w_gu"][t]))
            _err(f"tenant {t} block {b} grad wg", gg, GB["wg"], tol, worst)
            _err(f"tenant {t} block {b} grad wu", gu, GB["wu"], tol, worst)
    print(f"largest max|err|/rms {worst[0]:.4e} (bound {tol})")


# chunk 1, 8 and 16: one 16-row query tile (four key slices per warp
# group); 24: two tiles; 40: three (one warp idle); 64: four, the longest.
@pytest.mark.parametrize("dm,C,D", [(256, 8, 7), (512, 16, 14), (256, 24, 7), (256, 40, 5),
                                    (256, 64, 3), (256, 1, 2)])
def test_flow_train_step_vs_oracle(dm, C, D):
    s = FlowSetup(dm=dm, F=dm, C=C, D=D)
    plan = s.plan()
    hidden = (torch.randn(plan.n_tokens, 256, generator=torch.Generator().manual_seed(1))
              .to(torch.bfloat16).cuda())
    inp = _inputs(plan, C, D)
    g, vel, loss, ws = s.run(plan, hidden, inp)
    # bf16 operands of every projection and of the attention inputs, fp32
    # residual stream and attention, two blocks: a few 2^-9 roundings per
    # block; a wrong term or index is off by O(1)
    _check(s, plan, hidden, inp, vel, loss, FLOW_GRAD_TOL)


def test_flow_bench_size_sampled_tenant_vs_oracle():
    """The launch configuration the flow bench times: 8 tenants x 4 samples
    (one 256-row image + 16..64 text rows each) on 2048-wide context rows,
    experts of width 1024, 4 blocks, SwiGLU 4096, chunk 16 x 32.  The whole
    group runs; one seeded tenant's velocities, loss and every parameter
    gradient are checked against the oracle."""
    import bench
    w, dims = bench.flow_workload(8, 4)
    fe = bench.FLOW_EXPERT
    s = FlowSetup(dm=fe["d_model"], F=fe["d_ff"], nb=fe["n_blocks"], C=fe["chunk"],
                  D=fe["action_dim"], d=dims["d_in"], seed=43, std=0.02, workload=w)
    plan = s.plan()
    hidden = (torch.randn(plan.n_tokens, dims["d_in"], generator=torch.Generator().manual_seed(9))
              .to(torch.bfloat16).cuda())
    inp = synth.make_flow_inputs(plan.n_samples, s.C, s.D, 44, device="cuda")
    g, vel, loss, ws = s.run(plan, hidden, inp)
    assert torch.isfinite(vel).all() and torch.isfinite(loss[:8]).all()
    t = int(np.random.default_rng(5).integers(8))
    _check(s, plan, hidden, inp, vel, loss, FLOW_GRAD_TOL, only={t})


def test_flow_sampling_vs_oracle():
    s = FlowSetup()
    plan = s.plan()
    hidden = (torch.randn(plan.n_tokens, 256, generator=torch.Generator().manual_seed(2))
              .to(torch.bfloat16).cuda())
    noise = torch.randn(plan.n_samples, s.C, s.D, generator=torch.Generator().manual_seed(3)).cuda()
    g = R.DeviceGroup(plan)
    ws = torch.zeros(max(s.heads.workspace_bytes(g), 256), dtype=torch.uint8, device="cuda")
    out = torch.full_like(noise, float("nan"))
    s.heads.sample(g, hidden, noise, 4, out, ws)
    torch.cuda.synchronize()
    H = f64(hidden)
    cu, seg = plan.cu_seqlens, plan.seg_offsets
    for gi, t in enumerate(plan.slot_tenant.tolist()):
        p = s.oracle_params(t)
        for i in range(seg[gi], seg[gi + 1]):
            ref = Fl.sample(p, s.nh, H[cu[i]:cu[i + 1]], f64(noise[i]), 4)
            e = rel_err(f64(out[i]), ref)
            print(f"tenant {t} sample {i} Euler sample: max|err|/rms {e:.4e}")
            assert e < BF16_TOL, (t, i, e)


def test_flow_grouped_equals_isolated_and_other_slots_untouched():
    s = FlowSetup()
    plan = s.plan()
    hidden = (torch.randn(plan.n_tokens, 256, generator=torch.Generator().manual_seed(5))
              .to(torch.bfloat16).cuda())
    inp = _inputs(plan, s.C, s.D)
    _, vel, loss, _ = s.run(plan, hidden, inp)
    full = {k: v.clone() for k, v in s.heads.grads.items()}
    fullb = [{k: v.clone() for k, v in g.items()} for g in s.heads.block_grads]
    for v in list(s.heads.grads.values()) + [v for g in s.heads.block_grads for v in g.values()]:
        v.fill_(7.0)
    # tenant 2 alone: its samples, rows and inputs cut out of the group's
    t = 2
    gi = plan.slot_tenant.tolist().index(t)
    s0, s1 = plan.seg_offsets[gi], plan.seg_offsets[gi + 1]
    sub = s.plan([t])
    r0, r1 = plan.cu_seqlens[s0], plan.cu_seqlens[s1]
    inp1 = {k: v[s0:s1].contiguous() for k, v in inp.items()}
    _, vel1, loss1, _ = s.run(sub, hidden[r0:r1].contiguous(), inp1)
    assert torch.equal(vel1, vel[s0:s1])
    assert float(loss1[t]) == float(loss[t])
    for k, v in s.heads.grads.items():
        assert torch.equal(v[t], full[k][t]), k
        for u in range(3):
            if u != t:
                assert torch.all(v[u] == 7.0), (k, u)
    for b, g in enumerate(s.heads.block_grads):
        for k, v in g.items():
            assert torch.equal(v[t], fullb[b][k][t]), (b, k)
            assert torch.all(v[0] == 7.0) and torch.all(v[1] == 7.0), (b, k)


def test_flow_gradient_accumulation():
    s = FlowSetup(nb=1)
    plan = s.plan()
    hidden = (torch.randn(plan.n_tokens, 256, generator=torch.Generator().manual_seed(6))
              .to(torch.bfloat16).cuda())
    inp = _inputs(plan, s.C, s.D)
    s.run(plan, hidden, inp)
    one = {k: v.clone() for k, v in s.heads.grads.items()}
    oneb = [{k: v.clone() for k, v in g.items()} for g in s.heads.block_grads]
    s.run(plan, hidden, inp, accumulate=True)
    for k, v in s.heads.grads.items():
        assert torch.equal(v, 2 * one[k]), k
    for b, g in enumerate(s.heads.block_grads):
        for k, v in g.items():
            assert torch.equal(v, 2 * oneb[b][k]), (b, k)


def test_flow_rejects_bad_dimensions():
    s = FlowSetup()
    plan = s.plan()
    g = R.DeviceGroup(plan)
    s.heads.struct.d_model = 384  # not a supported width
    hidden = torch.zeros(plan.n_tokens, 256, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    inp = _inputs(plan, s.C, s.D)
    vel = torch.zeros(plan.n_samples, s.C, s.D, device="cuda")
    loss = torch.zeros(3, device="cuda")
    with pytest.raises(J.JnxError):
        s.heads.forward(g, hidden, inp["actions"], inp["noise"], inp["tau"], vel, loss, ws)


def test_flow_rejects_misaligned_workspace():
    s = FlowSetup()
    plan = s.plan()
    g = R.DeviceGroup(plan)
    hidden = torch.zeros(plan.n_tokens, 256, dtype=torch.bfloat16, device="cuda")
    ws = torch.zeros(max(s.heads.workspace_bytes(g), 256) + 512, dtype=torch.uint8, device="cuda")
    inp = _inputs(plan, s.C, s.D)
    vel = torch.full((plan.n_samples, s.C, s.D), -3.0, device="cuda")
    loss = torch.full((3,), -3.0, device="cuda")
    with pytest.raises(J.JnxError, match="aligned"):
        s.heads.forward(g, hidden, inp["actions"], inp["noise"], inp["tau"], vel, loss, ws[16:])
    torch.cuda.synchronize()
    assert torch.all(vel == -3.0) and torch.all(loss == -3.0)  # rejected before any launch
