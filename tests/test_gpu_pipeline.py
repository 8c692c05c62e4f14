"""Whole-path parity through the C ABI: plan -> backbone -> heads forward ->
loss -> heads backward, against the oracle's per-sample definition; grouped
vs per-tenant isolated on the GPU; slot isolation."""
import numpy as np
import pytest
import torch

import synth
from oracle import model as M
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.gpu_helpers import f64
from tests.helpers import BF16_TOL, GROUPED_TOL, deep_tol, grad_tols, oracle_requests, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


class Setup:
    """Everything a grouped step needs on the device for one workload."""

    def __init__(self, w, std=0.02, tenants=None, gen_device="cpu"):
        self.w = w
        self.bw = synth.make_backbone_weights(w, device=gen_device, std=std)
        self.hw = synth.make_head_weights(w, device=gen_device, std=std)
        self.inp = synth.make_inputs(w, device=gen_device)
        cuda = lambda t: t.cuda()
        self.bw_d = dict(layers=[{k: cuda(v) for k, v in L.items()} for L in self.bw["layers"]],
                         final_norm=cuda(self.bw["final_norm"]),
                         text_table=cuda(self.bw["text_table"]))
        self.hw_d = [{k: cuda(v) for k, v in h.items()} for h in self.hw]
        self.inp_d = {k: cuda(v) for k, v in self.inp.items()}
        self.bb = R.DeviceBackbone(w.backbone, self.bw_d, n_tenants=len(w.tenants))
        self.heads = R.DeviceHeads(w.tenants, w.backbone.d, self.hw_d)

    def run(self, wsub=None):
        w = wsub or self.w
        plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                                w.max_tokens)
        g = R.DeviceGroup(plan)
        step = R.GroupedStep(self.bb, self.heads, g)
        preds = torch.full_like(self.inp_d["targets"], float("nan"))
        step.run(self.inp_d["vision"], self.inp_d["text_ids"], self.inp_d["targets"], preds)
        R.check_status(step.ws_bb)
        R.check_status(step.ws_h)
        torch.cuda.synchronize()
        return plan, step, preds

    def oracle(self, tenants=None, n_layers=None):
        np_bw = synth.to_numpy_tree(self.bw)
        if self.w.backbone.d * self.w.backbone.d_ff * self.w.backbone.n_layers < 5e8:
            np_bw = M.widen_tree(np_bw)
        return M.grouped_step(self.w, np_bw, synth.to_numpy_tree(self.hw),
                              synth.to_numpy_tree(self.inp), tenants=tenants, n_layers=n_layers)


def _packed_index(plan, w):
    """Packed sample index of every (tenant, k-th sample of that tenant)."""
    out = {}
    seg = plan.seg_offsets
    for g, t in enumerate(plan.slot_tenant.tolist()):
        out[t] = list(range(seg[g], seg[g + 1]))
    return out


def _compare(setup, plan, step, preds, ref, tol=BF16_TOL, propagate_grads=False):
    w = setup.w
    idx = _packed_index(plan, w)
    loss = step.loss.cpu().numpy()
    for t, r in ref.items():
        feats = np.stack(r["feats"])
        got = f64(step.pooled[idx[t]])
        assert rel_err(got, feats) < tol, ("features", t, rel_err(got, feats))
        assert abs(loss[t] - r["loss"]) / abs(r["loss"]) < tol, ("loss", t)
        samples = [s for q in w.requests if q.tenant == t for s in q.samples]
        P = np.stack([f64(preds[s.target_off:s.target_off + w.tenants[t].width])
                      for s in samples])
        assert rel_err(P, r["pred"]) < tol, ("pred", t, rel_err(P, r["pred"]))
        T = np.stack([setup.inp["targets"][s.target_off:s.target_off + w.tenants[t].width]
                      .double().cpu().numpy() for s in samples])
        gt = (grad_tols(w.tenants[t].head_kind, M.widen_tree(synth.to_numpy_tree(setup.hw[t])),
                        r["feats"], T, tol) if propagate_grads
              else {k: tol for k in r["grads"]})
        for k, gref in r["grads"].items():
            e = rel_err(f64(setup.heads.grads[t][k]), gref)
            assert e < gt[k], ("grad", t, k, e, gt[k])


def test_tiny_full_group_vs_oracle():
    s = Setup(synth.make_workload("tiny"))
    plan, step, preds = s.run()
    _compare(s, plan, step, preds, s.oracle())


def test_tiny_sharp_attention_vs_oracle():
    s = Setup(synth.make_workload("tiny", qk_std=0.2))
    plan, step, preds = s.run()
    _compare(s, plan, step, preds, s.oracle())


def test_small_vs_oracle_on_whole_tenants():
    w = synth.make_workload("small")
    s = Setup(w)
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t) for t in range(8)}
    pick = sorted(counts, key=lambda t: counts[t])[:2]   # the two smallest tenants
    _compare(s, plan, step, preds, s.oracle(tenants=pick))


def test_grouped_equals_isolated_on_gpu():
    w = synth.make_workload("small")
    s = Setup(w)
    plan, step, preds = s.run()
    full_pooled = step.pooled.clone()
    full_loss = step.loss.clone()
    full_grads = [{k: v.clone() for k, v in g.items()} for g in s.heads.grads]
    idx = _packed_index(plan, w)
    for t in (0, 3, 6):
        p1, st1, pr1 = s.run(w.subset([t]))
        got = f64(st1.pooled[:len(idx[t])])
        assert rel_err(got, f64(full_pooled[idx[t]])) <= GROUPED_TOL
        assert abs(float(st1.loss[t]) - float(full_loss[t])) <= GROUPED_TOL * abs(float(full_loss[t]))
        for k in full_grads[t]:
            assert rel_err(f64(s.heads.grads[t][k]), f64(full_grads[t][k])) <= GROUPED_TOL
        # reported: bit-identical in practice (same kernels, same reduction order)
        assert torch.equal(st1.pooled[:len(idx[t])], full_pooled[idx[t]])


def test_slots_outside_the_group_are_not_touched():
    w = synth.make_workload("small")
    s = Setup(w)
    for g in s.heads.grads:
        for v in g.values():
            v.fill_(12345.0)
    sub = w.subset([1, 4])
    plan, step, preds = s.run(sub)
    for t in range(8):
        for k, v in s.heads.grads[t].items():
            untouched = bool(torch.all(v == 12345.0))
            assert untouched == (t not in (1, 4)), (t, k)
    loss = step.loss.cpu().numpy()
    assert all(np.isnan(loss[t]) for t in range(8) if t not in (1, 4))


def test_other_tenants_targets_do_not_change_a_tenants_grads():
    w = synth.make_workload("tiny")
    s = Setup(w)
    s.run()
    g0 = {k: v.clone() for k, v in s.heads.grads[0].items()}
    tb = [q for q in w.requests if q.tenant == 1][0].samples
    for smp in tb:
        s.inp_d["targets"][smp.target_off:smp.target_off + 56] += 0.75
    s.run()
    for k in g0:
        assert torch.equal(g0[k], s.heads.grads[0][k])


@pytest.mark.slow
def test_llama7b_full_size_sampled_sample():
    """The 7B-class workload at full size (~65.8k packed tokens, 32 blocks)
    in the benchmark's launch configuration; the shortest sample's pooled
    feature is checked against the oracle's per-sample forward."""
    w = synth.make_workload("llama7b")
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    assert torch.isfinite(step.pooled).all() and torch.isfinite(step.loss[:32]).all()
    L = np.diff(plan.cu_seqlens)
    si = int(np.argmin(L))
    # which arrival-order sample is packed sample si
    order = [smp for t in plan.slot_tenant.tolist() for q in w.requests if q.tenant == t
             for smp in q.samples]
    smp = order[si]
    bb = M.backbone_dict(w)
    np_bw = synth.to_numpy_tree(s.bw)
    npi = synth.to_numpy_tree(s.inp)
    x = M.sample_embeddings(bb, vars(smp), npi["vision"], npi["text_ids"], np_bw["text_table"])
    ref = M.mean_pool(M.backbone_sample(bb, np_bw, x))
    e = rel_err(f64(step.pooled[si]), ref)
    assert e < deep_tol(w.backbone.n_layers), e


def test_llama7b_shapes_one_block_whole_tenants():
    """Every kernel at the 7B-class widths and the full packed length
    (~65.8k tokens, 32 tenants), one block deep so the stated 2e-2 bound
    applies to the whole path; the two smallest tenants are checked end to
    end (features, loss, predictions, head gradients)."""
    w = synth.make_workload("llama7b", n_layers=1)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t) for t in range(32)}
    pick = sorted(counts, key=lambda t: (counts[t], t))[:2]
    _compare(s, plan, step, preds, s.oracle(tenants=pick), propagate_grads=True)


@pytest.mark.parametrize("name", ["small", "llama7b"])
def test_heads_stage_on_synthetic_features(name):
    """The head stage alone at the workload's head shapes, on seeded random
    pooled features (inputs from the generator, not from the backbone)."""
    w = synth.make_workload(name)
    hw = synth.make_head_weights(w)
    inp = synth.make_inputs(w)
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    pooled = torch.randn((plan.n_samples, w.backbone.d),
                         generator=torch.Generator().manual_seed(3)).cuda()
    heads = R.DeviceHeads(w.tenants, w.backbone.d, [{k: v.cuda() for k, v in h.items()} for h in hw])
    ws = torch.zeros(heads.workspace_bytes(g), dtype=torch.uint8, device="cuda")
    tg = inp["targets"].cuda()
    preds = torch.full_like(tg, float("nan"))
    loss = torch.full((len(w.tenants),), float("nan"), device="cuda")
    heads.forward(g, pooled, None, tg, preds, loss, ws)
    heads.backward(g, pooled, None, tg, ws)
    torch.cuda.synchronize()
    P = f64(pooled)
    npT = synth.to_numpy_tree(inp)["targets"]
    seg = plan.seg_offsets
    for gi, t in enumerate(plan.slot_tenant.tolist()):
        tn = w.tenants[t]
        samples = [s for q in w.requests if q.tenant == t for s in q.samples]
        T = np.stack([npT[s.target_off:s.target_off + tn.width] for s in samples])
        feats = list(P[seg[gi]:seg[gi + 1]])
        lo, Y, gr = M.tenant_step(0, synth.to_numpy_tree(hw[t]), feats, T)
        assert abs(float(loss[t]) - lo) < 1e-4 * abs(lo)
        got = np.stack([f64(preds[s.target_off:s.target_off + tn.width]) for s in samples])
        assert rel_err(got, Y) < 1e-4
        for k, v in gr.items():
            e = rel_err(f64(heads.grads[t][k]), v)
            assert e < 1e-4, (t, k, e)


@pytest.mark.parametrize("nq,dq", [(32, 256), (8, 512)])
def test_query_heads_stage_on_synthetic_hidden_rows(nq, dq):
    """The cross-attention query head alone (2B-class head shapes: 32 queries
    x 256, and 8 queries x 512 for the wide-query path with two value-column
    passes; d = 2048, widths 350 / 700 / 1600) on seeded random hidden rows,
    for three tenants of the MQA workload, against the oracle."""
    import dataclasses
    w = synth.make_workload("mqa2b").subset([0, 1, 2])
    w = dataclasses.replace(w, tenants=[dataclasses.replace(tn, n_queries=nq, q_dim=dq)
                                        for tn in w.tenants])
    hw = synth.make_head_weights(w)
    inp = synth.make_inputs(w)
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), 1 << 30, 1 << 30)
    g = R.DeviceGroup(plan)
    X = (torch.randn((plan.n_tokens, w.backbone.d), generator=torch.Generator().manual_seed(5))
         .to(torch.bfloat16).cuda())
    heads = R.DeviceHeads(w.tenants, w.backbone.d, [{k: v.cuda() for k, v in h.items()} for h in hw])
    ws = torch.zeros(heads.workspace_bytes(g), dtype=torch.uint8, device="cuda")
    tg = inp["targets"].cuda()
    preds = torch.full_like(tg, float("nan"))
    loss = torch.full((len(w.tenants),), float("nan"), device="cuda")
    heads.forward(g, None, X, tg, preds, loss, ws)
    heads.backward(g, None, X, tg, ws)
    torch.cuda.synchronize()
    Xn = f64(X)
    npT = synth.to_numpy_tree(inp)["targets"]
    cu = plan.cu_seqlens
    seg = plan.seg_offsets
    for gi, t in enumerate(plan.slot_tenant.tolist()):
        tn = w.tenants[t]
        samples = [s for q in w.requests if q.tenant == t for s in q.samples]
        T = np.stack([npT[s.target_off:s.target_off + tn.width] for s in samples])
        feats = [Xn[cu[i]:cu[i + 1]] for i in range(seg[gi], seg[gi + 1])]
        lo, Y, gr = M.tenant_step(1, M.widen_tree(synth.to_numpy_tree(hw[t])), feats, T)
        assert abs(float(loss[t]) - lo) < 1e-4 * abs(lo)
        got = np.stack([f64(preds[s.target_off:s.target_off + tn.width]) for s in samples])
        assert rel_err(got, Y) < 1e-4
        for k, v in gr.items():
            e = rel_err(f64(heads.grads[t][k]), v)
            assert e < 1e-3, (t, k, e)


def test_mqa2b_two_blocks_one_tenant_vs_oracle():
    """The 2B-class backbone (MQA 8 x 256 with one KV head, GeGLU 16384,
    1-3 images per sample) two blocks deep over the full 16-tenant packed
    batch (~137k tokens), with cross-attention query heads; the smallest
    tenant is checked end to end."""
    w = synth.make_workload("mqa2b", n_layers=2)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(smp.length(256) for r in w.requests if r.tenant == t for smp in r.samples)
              for t in range(len(w.tenants))}
    pick = [min(counts, key=lambda t: (counts[t], t))]
    ref = s.oracle(tenants=pick)
    t = pick[0]
    idx = _packed_index(plan, w)[t]
    cu = plan.cu_seqlens
    Hg = f64(step.hidden)
    for k, i in enumerate(idx):
        e = rel_err(Hg[cu[i]:cu[i + 1]], ref[t]["feats"][k])
        # hidden rows are stored in bf16: measure beyond that rounding
        from tests.helpers import rel_err_bf16_out
        e = rel_err_bf16_out(Hg[cu[i]:cu[i + 1]], ref[t]["feats"][k])
        assert e < BF16_TOL, ("hidden", k, e)
    loss = float(step.loss[t])
    assert abs(loss - ref[t]["loss"]) / abs(ref[t]["loss"]) < BF16_TOL
    samples = [smp for q in w.requests if q.tenant == t for smp in q.samples]
    P = np.stack([f64(preds[smp.target_off:smp.target_off + w.tenants[t].width]) for smp in samples])
    assert rel_err(P, ref[t]["pred"]) < BF16_TOL
    T = np.stack([s.inp["targets"][smp.target_off:smp.target_off + w.tenants[t].width]
                  .double().cpu().numpy() for smp in samples])
    gt = grad_tols(1, M.widen_tree(synth.to_numpy_tree(s.hw[t])), ref[t]["feats"], T, BF16_TOL)
    for k, gref in ref[t]["grads"].items():
        e = rel_err(f64(s.heads.grads[t][k]), gref)
        assert e < gt[k], ("grad", k, e, gt[k])


def test_lora_with_zero_up_projection_changes_nothing():
    """Per-tenant LoRA whose B matrices are zero must leave the backbone's
    output bit-identical to the same backbone without adapters."""
    import dataclasses
    w = synth.make_workload("zipf2b", n_layers=1)
    s = Setup(w, gen_device="cuda")
    for L in s.bw_d["layers"]:
        for p in ("q", "k", "v", "o"):
            L["lora_b_" + p].zero_()
    plan, step, preds = s.run()
    h_lora = step.hidden.clone()
    w0 = dataclasses.replace(w, backbone=dataclasses.replace(w.backbone, lora_rank=0))
    bb0 = R.DeviceBackbone(w0.backbone, s.bw_d, n_tenants=len(w.tenants))
    g = R.DeviceGroup(plan)
    hid = torch.zeros_like(h_lora)
    ws = torch.zeros(bb0.workspace_bytes(plan.n_tokens), dtype=torch.uint8, device="cuda")
    bb0.forward(g, s.inp_d["vision"], s.inp_d["text_ids"], None, hid, ws)
    torch.cuda.synchronize()
    assert torch.equal(hid, h_lora)


def test_zipf2b_lora_two_blocks_vs_oracle():
    """The skewed 64-tenant workload (Zipf counts, lengths 260..840, LoRA
    rank 16 on Q/K/V/O) two blocks deep over the full packed batch
    (~307k tokens); the two smallest tenants and the largest single-sample
    tenant are checked end to end against the oracle."""
    w = synth.make_workload("zipf2b", n_layers=2)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t)
              for t in range(len(w.tenants))}
    pick = sorted(counts, key=lambda t: (counts[t], t))[:2]
    ref = s.oracle(tenants=pick)
    idx = _packed_index(plan, w)
    cu = plan.cu_seqlens
    Hg = f64(step.hidden)
    from tests.helpers import rel_err_bf16_out
    for t in pick:
        for k, i in enumerate(idx[t]):
            e = rel_err_bf16_out(Hg[cu[i]:cu[i + 1]], ref[t]["feats"][k])
            assert e < BF16_TOL, ("hidden", t, k, e)
        assert abs(float(step.loss[t]) - ref[t]["loss"]) / abs(ref[t]["loss"]) < BF16_TOL
        samples = [smp for q in w.requests if q.tenant == t for smp in q.samples]
        P = np.stack([f64(preds[smp.target_off:smp.target_off + w.tenants[t].width])
                      for smp in samples])
        assert rel_err(P, ref[t]["pred"]) < BF16_TOL
        T = np.stack([s.inp["targets"][smp.target_off:smp.target_off + w.tenants[t].width]
                      .double().cpu().numpy() for smp in samples])
        gt = grad_tols(1, M.widen_tree(synth.to_numpy_tree(s.hw[t])), ref[t]["feats"], T,
                       BF16_TOL)
        for k, gref in ref[t]["grads"].items():
            e = rel_err(f64(s.heads.grads[t][k]), gref)
            assert e < gt[k], ("grad", t, k, e, gt[k])


def test_step_pipeline_matches_plain_steps():
    # StepPipeline overlaps each step's planning and input copy with the step
    # before it; every step must still give exactly what a plain step gives
    # (same kernels, same order), including a step whose group (one tenant)
    # differs from the previous one's
    w = synth.make_workload("tiny")
    s = Setup(w)
    _, ref_step, ref_preds = s.run()
    ref_loss = ref_step.loss.cpu()
    ref_preds = ref_preds.cpu()
    wsub = w.subset([0])
    sub_plan, sub_step, _ = s.run(wsub)
    sub_loss = sub_step.loss.cpu()

    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                            w.max_tokens)
    step = R.GroupedStep(s.bb, s.heads, R.DeviceGroup(plan))
    host = {k: v.cpu().pin_memory() for k, v in s.inp.items()}
    pipe = R.StepPipeline(step, s.inp["vision"].shape[0], s.inp["text_ids"].numel(),
                          tuple(s.inp["targets"].shape))
    order = ["full", "full", "sub", "full"]

    def plan_fn(i):
        ww = wsub if order[i] == "sub" else w
        return J.jnx_group_plan(ww.schemas(), oracle_requests(ww), len(w.tenants),
                                w.max_samples, w.max_tokens)

    got = {}
    pipe.run([host] * len(order), plan_fn,
             on_result=lambda i, loss, preds: got.__setitem__(i, (loss.clone(), preds.clone())))
    R.check_status(step.ws_bb)
    R.check_status(step.ws_h)
    assert sorted(got) == list(range(len(order)))
    for i, kind in enumerate(order):
        loss, preds = got[i]
        if kind == "full":
            assert torch.equal(loss, ref_loss), i
            assert torch.equal(preds, ref_preds), i
        else:
            for t in set(sub_plan.slot_tenant.tolist()):
                assert torch.equal(loss[t], sub_loss[t]), (i, t)


def test_inference_path_matches_training_forward_and_is_grouping_invariant():
    # the inference step (backbone + head forward, no targets) predicts what
    # the training step's forward predicts, and a tenant's predictions are
    # the same in the group as alone (bit for bit: same kernels, same order)
    w = synth.make_workload("small")
    s = Setup(w)
    plan, step, preds_train = s.run()
    preds = torch.full_like(preds_train, float("nan"))
    step.infer(s.inp_d["vision"], s.inp_d["text_ids"], preds)
    R.check_status(step.ws_bb)
    torch.cuda.synchronize()
    assert torch.equal(preds, preds_train)
    for t in (0, 5):
        wsub = w.subset([t])
        p1 = J.jnx_group_plan(wsub.schemas(), oracle_requests(wsub), len(w.tenants),
                              w.max_samples, w.max_tokens)
        st1 = R.GroupedStep(s.bb, s.heads, R.DeviceGroup(p1))
        pr1 = torch.full_like(preds, float("nan"))
        st1.infer(s.inp_d["vision"], s.inp_d["text_ids"], pr1)
        torch.cuda.synchronize()
        offs = [int(o) for o in p1.sample_target]
        width = w.tenants[t].width
        for o in offs:
            assert torch.equal(pr1.view(-1)[o:o + width], preds.view(-1)[o:o + width]), (t, o)


@pytest.mark.filterwarnings("ignore:The CUDA Graph is empty")
def test_backbone_forward_without_a_device_work_list_refuses_graph_capture():
    """Without the group's device copy of the attention work list the
    backbone forward uploads it from host memory, which a CUDA graph would
    replay from a freed buffer: a capturing stream is refused before any
    launch (nothing is replayed here), and the step still runs eagerly."""
    s = Setup(synth.make_workload("tiny"))
    plan, step, preds = s.run()
    step.group.struct.attn_items = None
    step.group.struct.n_attn_items = 0
    stream = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with pytest.raises(J.JnxError, match="CUDA graph"):
        with torch.cuda.graph(graph, stream=stream):
            step.run(s.inp_d["vision"], s.inp_d["text_ids"], s.inp_d["targets"], preds)
    del graph
    torch.cuda.synchronize()
    preds2 = torch.full_like(preds, float("nan"))
    step.run(s.inp_d["vision"], s.inp_d["text_ids"], s.inp_d["targets"], preds2)
    torch.cuda.synchronize()
    assert torch.equal(preds2, preds)


@pytest.mark.parametrize("name", ["tiny", "mqa2b"])
def test_grouped_step_replays_as_a_cuda_graph(name):
    """With the group's work list on the device the whole grouped step
    (backbone, heads forward, loss, heads backward) is captured once and
    replayed; the replay gives the eager step's predictions, losses and head
    gradients bit for bit."""
    w = synth.make_workload(name, n_layers=1) if name != "tiny" else synth.make_workload(name)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    want_p, want_l = preds.clone(), step.loss.clone()
    want_g = [{k: v.clone() for k, v in g.items()} for g in s.heads.grads]
    stream = torch.cuda.Stream()
    stream.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step.run(s.inp_d["vision"], s.inp_d["text_ids"], s.inp_d["targets"], preds)
    preds.fill_(float("nan"))
    for g in s.heads.grads:
        for v in g.values():
            v.fill_(7.0)
    graph.replay()
    torch.cuda.synchronize()
    R.check_status(step.ws_bb)
    R.check_status(step.ws_h)
    assert torch.equal(preds, want_p) and torch.equal(step.loss, want_l)
    for g, wg in zip(s.heads.grads, want_g):
        for k in g:
            assert torch.equal(g[k], wg[k]), k
