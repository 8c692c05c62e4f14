"""Helpers for GPU tests: seeded test tensors and conversions for the oracle."""
import numpy as np
import torch

import synth
from oracle import model as M
from paper_2607_16074_gb300 import jnx as J
from paper_2607_16074_gb300 import runtime as R
from tests.helpers import SAMPLE_FLOOR_FACTOR, gate, oracle_requests, rel_err


def dev():
    return torch.device("cuda")


def randn_bf16(shape, seed, std=1.0, device="cuda"):
    g = torch.Generator().manual_seed(seed)
    return (torch.randn(*shape, generator=g) * std).to(torch.bfloat16).to(device)


def f64(t):
    """A torch tensor (any dtype, any device) as a float64 numpy array (exact
    for bf16/fp32)."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def ptr(t):
    return t.data_ptr()


def stream():
    return torch.cuda.current_stream().cuda_stream


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


def packed_index(plan, w):
    """Packed sample indices of every tenant's samples (in arrival order)."""
    out = {}
    seg = plan.seg_offsets
    for g, t in enumerate(plan.slot_tenant.tolist()):
        out[t] = list(range(seg[g], seg[g + 1]))
    return out


def tenant_samples(w, t):
    """Tenant t's samples in arrival order."""
    return [smp for q in w.requests if q.tenant == t for smp in q.samples]


def oracle_and_floor(setup, pick):
    """For every sample of the tenants in pick: the oracle's features (its
    per-sample forward, oracle.model.block one layer at a time) and the
    emulated features with every rounding point of the CUDA path
    (tests/bf16_emulation.py), on the same inputs; each layer's weights are
    widened once for all samples.  Pooled features for MLP-head tenants,
    final normed rows for query-head tenants."""
    from tests import bf16_emulation as E
    w = setup.w
    np_bw = synth.to_numpy_tree(setup.bw)
    npi = synth.to_numpy_tree(setup.inp)
    bb = M.backbone_dict(w)
    samples = [(t, smp) for t in pick for smp in tenant_samples(w, t)]
    xs = [M.sample_embeddings(bb, vars(smp), npi["vision"], npi["text_ids"], np_bw["text_table"])
          for _, smp in samples]
    tenants = [t for t, _ in samples]
    emu = E.Emulation(w.backbone, xs, tenants, E.ALL)
    ref = list(xs)
    for lw in np_bw["layers"]:
        wl = E.widen_layer(lw)
        ref = [M.block(bb, wl, x, t) for x, t in zip(ref, tenants)]
        emu.block(wl)
    fin = np_bw["final_norm"]
    ref = [M.rmsnorm(x, fin, bb["eps"]) for x in ref]
    em_rows, em_pool = emu.final(fin), emu.pooled(fin)
    out = {t: dict(ref=[], emu=[]) for t in pick}
    for (t, _), r, er, ep in zip(samples, ref, em_rows, em_pool):
        mlp = w.tenants[t].head_kind == synth.HEAD_MLP
        out[t]["ref"].append(M.mean_pool(r) if mlp else r)
        out[t]["emu"].append(ep if mlp else er)
    return out


def check_tenants(name, setup, plan, step, preds, pick):
    """Whole-path parity of every tenant in pick against the oracle, in the
    stated measure max|err|/rms(ref) (nothing subtracted), each quantity
    gated by gate(floor): the stated 2e-2, or FLOOR_FACTOR times the floor
    that the CUDA path's own roundings set (the emulated forward's distance
    from the oracle, and the oracle's head step on the emulated features).
    Checks each tenant's features (pooled, or final normed rows for a query
    head) as a whole and every sample's (at SAMPLE_FLOOR_FACTOR), each
    tenant's predictions, loss and head gradients; prints every number.
    Returns the largest ratio of GPU error to floor at FLOOR_FACTOR gates."""
    w = setup.w
    feats = oracle_and_floor(setup, pick)
    idx = packed_index(plan, w)
    cu = plan.cu_seqlens
    pooled = f64(step.pooled) if step.pooled is not None else None
    hid = f64(step.hidden) if step.hidden is not None else None
    loss = step.loss.cpu().numpy()
    worst = 0.0

    def one(what, e, fl, factor=None):
        nonlocal worst
        gt = gate(fl) if factor is None else gate(fl, factor)
        if factor is None:
            worst = max(worst, e / max(fl, 1e-300))
        print(f"{name} {what}: gpu {e:.4e}  floor {fl:.4e}  ratio {e / max(fl, 1e-300):.3f}  "
              f"gate {gt:.4e}")
        assert e <= gt, (name, what, e, fl)

    for t in pick:
        tn = w.tenants[t]
        mlp = tn.head_kind == synth.HEAD_MLP
        samples = tenant_samples(w, t)
        kind = "pooled" if mlp else "rows"
        gs = [pooled[i] if mlp else hid[cu[i]:cu[i + 1]] for i in idx[t]]
        for k, g in enumerate(gs):
            r, e = feats[t]["ref"][k], feats[t]["emu"][k]
            one(f"tenant {t} sample {k} {kind}", rel_err(g, r), rel_err(e, r),
                SAMPLE_FLOOR_FACTOR)
        cat = lambda xs: np.concatenate([np.ravel(x) for x in xs])
        R_, E_ = cat(feats[t]["ref"]), cat(feats[t]["emu"])
        one(f"tenant {t} all samples' {kind}", rel_err(cat(gs), R_), rel_err(E_, R_))
        hw = M.widen_tree(synth.to_numpy_tree(setup.hw[t]))
        T = np.stack([setup.inp["targets"][smp.target_off:smp.target_off + tn.width]
                      .double().cpu().numpy() for smp in samples])
        l_ref, y_ref, g_ref = M.tenant_step(tn.head_kind, hw, feats[t]["ref"], T)
        l_emu, y_emu, g_emu = M.tenant_step(tn.head_kind, hw, feats[t]["emu"], T)
        P = np.stack([f64(preds[smp.target_off:smp.target_off + tn.width]) for smp in samples])
        one(f"tenant {t} predictions", rel_err(P, y_ref), rel_err(y_emu, y_ref))
        one(f"tenant {t} loss (relative)", abs(float(loss[t]) - l_ref) / abs(l_ref),
            abs(l_emu - l_ref) / abs(l_ref))
        for key in g_ref:
            one(f"tenant {t} grad {key}", rel_err(f64(setup.heads.grads[t][key]), g_ref[key]),
                rel_err(g_emu[key], g_ref[key]))
    print(f"{name}: largest ratio of gpu error to floor {worst:.3f}")
    return worst
