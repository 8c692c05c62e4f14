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
from tests.gpu_helpers import Setup, check_tenants, f64, packed_index as _packed_index
from tests.helpers import GROUPED_TOL, oracle_requests, rel_err

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def _compare(setup, plan, step, preds, pick=None, name=""):
    """Whole tenants end to end against the oracle in the stated measure,
    each quantity gated by the stated 2e-2 or 1.3 x its bf16 floor
    (tests/gpu_helpers.py check_tenants)."""
    w = setup.w
    if pick is None:
        pick = sorted(set(plan.slot_tenant.tolist()))
    check_tenants(name or w.name, setup, plan, step, preds, pick)


def test_tiny_full_group_vs_oracle():
    s = Setup(synth.make_workload("tiny"))
    plan, step, preds = s.run()
    _compare(s, plan, step, preds)


def test_tiny_sharp_attention_vs_oracle():
    s = Setup(synth.make_workload("tiny", qk_std=0.2))
    plan, step, preds = s.run()
    _compare(s, plan, step, preds, name="tiny sharp")


def test_small_vs_oracle_on_whole_tenants():
    w = synth.make_workload("small")
    s = Setup(w)
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t) for t in range(8)}
    pick = sorted(counts, key=lambda t: counts[t])[:2]   # the two smallest tenants
    _compare(s, plan, step, preds, pick)


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


def test_empty_plan_and_zero_sizes_write_nothing():
    """Degenerate inputs: a GEMM of zero rows, attention over zero samples,
    and a whole grouped step (backbone, heads forward, loss, heads backward)
    over the plan of an empty request queue all return JNX_OK and leave
    every output as it was."""
    from tests.gpu_helpers import randn_bf16, stream
    L = J.lib()
    A = randn_bf16((1, 256), 1)
    W = randn_bf16((256, 256), 2, 0.05)
    out = torch.full((1, 256), 7.0, device="cuda")
    J.check(L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), 0, 256, 256, J.JNX_EPI_F32,
                          out.data_ptr(), 256, None, 0, 0, 0, 0.0, 0, None, 0, stream()))
    qkv = randn_bf16((1, 3 * 128), 3)
    o = torch.full((1, 128), 7.0, dtype=torch.bfloat16, device="cuda")
    cu = torch.zeros(1, dtype=torch.int32, device="cuda")
    J.check(L.jnx_op_attention(qkv.data_ptr(), 0, 1, 1, 128, cu.data_ptr(), 0, 0, o.data_ptr(),
                               None, stream()))
    w = synth.make_workload("tiny")
    s = Setup(w)
    plan = J.jnx_group_plan(w.schemas(), [], len(w.tenants), w.max_samples, w.max_tokens)
    assert plan.n_samples == 0 and plan.n_tokens == 0 and plan.n_slots == 0
    g = R.DeviceGroup(plan)
    step = R.GroupedStep(s.bb, s.heads, g)
    preds = torch.full_like(s.inp_d["targets"], 7.0)
    grads_before = [v.clone() for gr in s.heads.grads for v in gr.values()]
    step.run(s.inp_d["vision"], s.inp_d["text_ids"], s.inp_d["targets"], preds)
    R.check_status(step.ws_bb)
    R.check_status(step.ws_h)
    torch.cuda.synchronize()
    assert (out == 7).all() and (o == 7).all() and (preds == 7).all()
    for a, b in zip(grads_before, [v for gr in s.heads.grads for v in gr.values()]):
        assert torch.equal(a, b)


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


def test_llama7b_shapes_one_block_whole_tenants():
    """Every kernel at the 7B-class widths and the full packed length
    (~65.8k tokens, 32 tenants), one block deep; the two smallest tenants
    are checked end to end (features, loss, predictions, head gradients).
    The 32-block depth is checked in tests/test_gpu_full_depth.py."""
    w = synth.make_workload("llama7b", n_layers=1)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t) for t in range(32)}
    pick = sorted(counts, key=lambda t: (counts[t], t))[:2]
    _compare(s, plan, step, preds, pick, name="llama7b 1 block")


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
        e_y = rel_err(got, Y)
        e_g = {k: rel_err(f64(heads.grads[t][k]), v) for k, v in gr.items()}
        print(f"query head nq={nq} dq={dq} tenant {t}: preds {e_y:.2e}, grads "
              + ", ".join(f"{k} {e:.2e}" for k, e in e_g.items()))
        assert e_y < 1e-4
        for k, e in e_g.items():
            assert e < 1e-3, (t, k, e)


def test_mqa2b_two_blocks_one_tenant_vs_oracle():
    """The 2B-class backbone (MQA 8 x 256 with one KV head, GeGLU 16384,
    1-3 images per sample) two blocks deep over the full 16-tenant packed
    batch (~137k tokens), with cross-attention query heads; the smallest
    tenant is checked end to end (final normed rows of every sample,
    predictions, loss, head gradients)."""
    w = synth.make_workload("mqa2b", n_layers=2)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(smp.length(256) for r in w.requests if r.tenant == t for smp in r.samples)
              for t in range(len(w.tenants))}
    pick = [min(counts, key=lambda t: (counts[t], t))]
    _compare(s, plan, step, preds, pick, name="mqa2b 2 blocks")


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
    (~307k tokens); the two smallest tenants are checked end to end against
    the oracle."""
    w = synth.make_workload("zipf2b", n_layers=2)
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: sum(len(r.samples) for r in w.requests if r.tenant == t)
              for t in range(len(w.tenants))}
    pick = sorted(counts, key=lambda t: (counts[t], t))[:2]
    _compare(s, plan, step, preds, pick, name="zipf2b 2 blocks")


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
