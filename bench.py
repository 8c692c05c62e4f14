"""Benchmark of the grouped multi-tenant step on GB300.

One step = one pass of the whole hot path over one group: host plan (timed
separately), packer, all backbone blocks over the packed varlen batch,
final norm + pool, every tenant's head forward, L2 loss and head backward.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload llama7b]
    python bench.py --impl reference ...   # the fp64 CPU oracle, timed

Prints ONE JSON line (rank 0).  `value` is whole-job tokens/s with inputs
resident in HBM; `e2e` is the same metric through the C ABI with the step's
inputs copied from pinned host memory and its losses / predictions read back
inside the timed region.  With N > 1 (torchrun) every rank runs its own
group (independent replicas, weak scaling, no data-path collective).
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "grouped fwd+head-bwd tokens/s on 1 GB300; % bf16 tensor peak; speedup vs per-tenant"


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"],
                    bf16_sustained=d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                    source="measured")
    except Exception:
        return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


def workload_desc(w):
    b = w.backbone
    return (f"{w.name}: {len(w.tenants)} tenants, {len(w.samples)} samples, "
            f"{w.n_tokens} packed tokens; {b.n_layers} blocks d={b.d} {b.n_heads}x{b.head_dim} "
            f"heads ({b.n_kv_heads} kv), FFN {b.d_ff} {'SwiGLU' if b.glu == 0 else 'GeGLU'}")


# DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) of one gate/up
# GEMM launch: captured by ncu on a small launch of the same kernel whose
# row blocks fill whole tile groups, as the full launch's do (10,240 rows),
# and scaled by rows to the full launch (the traffic per row is the same:
# A once, the weight once per tile group, u once; the summary and command
# are in profiles/).  Valid only for the GEMM source it was taken on and the
# launch shape it is scaled to (packed rows, width, FFN width).
RECORDED_TRAFFIC = {
    # workload: (sha256 of csrc/gemm.cu, (rows, d, F), bytes per launch, profile)
    "llama7b": ("8ae0084ca22eba83c00bdc18a9ece2d9956dbc2873b4f8142777cc187087ec5e",
                (65817, 4096, 11008), (465.714176e6 + 215.440640e6) * 65817 / 10240,
                "profiles/gemm_gate_up_glu_10240_dram.md (10,240 rows, scaled by rows)"),
}


def gemm_source_hash() -> str:
    import hashlib
    p = os.path.join(ROOT, "paper_2607_16074_gb300", "csrc", "gemm.cu")
    with open(p, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def recorded_traffic(workload: str, shape):
    """The recorded traffic of the gate/up launch, or None when the GEMM
    source or the launch shape (rows, d, F) differs from the capture's."""
    rec = RECORDED_TRAFFIC.get(workload)
    if not rec or rec[0] != gemm_source_hash() or tuple(rec[1]) != tuple(shape):
        return None
    return dict(bytes_per_launch=rec[2], source=rec[3])


def gu_algorithmic_bytes(w, n_tokens: int) -> int:
    """Bytes the gate/up GEMM must move at least: read the normed rows
    [N, d] and the fused gate/up weights [2F, d], write u [N, F] (bf16)."""
    b = w.backbone
    return int(2 * (n_tokens * b.d + 2 * b.d_ff * b.d + n_tokens * b.d_ff))


def replica_seed(base_seed: int, rank: int) -> int:
    """With N > 1 every rank runs its own independent group: the same shapes,
    its own seeded inputs and weights (no data-path collective)."""
    return base_seed + 1000 * rank


def max_over_ranks(value: float, world: int, device=None) -> float:
    """The job's time is its slowest rank's (barrier-bracketed region)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank: int, world: int, steps: int, t_ms: float) -> float:
    """Whole-job throughput: the tokens all ranks processed over the job time."""
    return tokens_per_rank * world * steps / (t_ms / 1e3)


def make_bench_workload(args):
    import synth
    over = {"n_layers": args.layers} if getattr(args, "layers", 0) else {}
    w = synth.make_workload(args.workload, **over)
    if getattr(args, "subset", 0):
        w = w.subset(list(range(args.subset)))
    return w


def oracle_requests(w):
    return [dict(tenant=r.tenant, schema=r.schema,
                 samples=[dict(n_img=s.n_img, text_len=s.text_len, vision_row=s.vision_row,
                               text_pos=s.text_pos, target_off=s.target_off) for s in r.samples])
            for r in w.requests]


# ---------------------------------------------------------------------------
# CPU oracle timing (the reference arm and the cpu_baseline key)
# ---------------------------------------------------------------------------

def oracle_tenant_subset(w):
    """The whole tenants the oracle timing covers: every tenant of the
    one- and six-block workloads, otherwise the two with the most tokens and
    the two with the fewest (ties by tenant index)."""
    v = w.backbone.vision_tokens
    tok = {}
    for r in w.requests:
        tok[r.tenant] = tok.get(r.tenant, 0) + sum(s.length(v) for s in r.samples)
    if w.name in ("tiny", "small"):
        return sorted(tok)
    order = sorted(tok, key=lambda t: (tok[t], t))
    return sorted(set(order[:2] + order[-2:]))


def oracle_tenant_run(w, tenants, n_layers, bw_np, hw_np, inp_np):
    """Time the fp64 oracle, as it stands, on whole tenants: every sample's
    backbone forward alone through n_layers blocks, final norm and pool
    (oracle.model.sample_features), then each tenant's head, loss and head
    gradients (oracle.model.tenant_step).  Returns the backbone seconds, the
    head seconds, the tokens and the samples timed."""
    from oracle import model as M
    bb = M.backbone_dict(w)
    tg = np.asarray(inp_np["targets"], dtype=np.float64)
    t_bb = t_head = 0.0
    toks = n = 0
    for t in tenants:
        tn = w.tenants[t]
        samples = [s for r in w.requests if r.tenant == t for s in r.samples]
        t0 = time.perf_counter()
        feats = [M.sample_features(bb, bw_np, vars(s), t, inp_np, tn.head_kind, n_layers)
                 for s in samples]
        t1 = time.perf_counter()
        T = np.stack([tg[s.target_off:s.target_off + tn.width] for s in samples])
        M.tenant_step(tn.head_kind, hw_np[t], feats, T)
        t2 = time.perf_counter()
        t_bb += t1 - t0
        t_head += t2 - t1
        toks += sum(s.length(w.backbone.vision_tokens) for s in samples)
        n += len(samples)
    return dict(backbone_s=t_bb, head_s=t_head, tokens=toks, samples=n)


def oracle_full_depth_s(w, r, n_layers):
    """Seconds the timed run would take at the workload's full depth: the
    backbone time scaled by blocks, the head time as measured."""
    return r["backbone_s"] * w.backbone.n_layers / n_layers + r["head_s"]


def host_numpy_inputs(w, bw, hw, inp, n_layers):
    """Host copies of what the oracle timing reads: the first n_layers blocks
    and the heads widened to fp64 once (outside the timed region, like
    loading weights), the text table and inputs as bf16 bit patterns."""
    import synth
    from oracle import model as M
    bw_np = dict(layers=[M.widen_tree(synth.to_numpy_tree(L)) for L in bw["layers"][:n_layers]],
                 final_norm=synth.bf16_bits(bw["final_norm"]),
                 text_table=synth.bf16_bits(bw["text_table"]))
    hw_np = [M.widen_tree(synth.to_numpy_tree(h)) for h in hw]
    return bw_np, hw_np, synth.to_numpy_tree(inp)


# ---------------------------------------------------------------------------
# clocks
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        # the raw samples (the JSON line carries their summary); JNX_BENCH_OUT
        # names another directory for them
        out = os.environ.get("JNX_BENCH_OUT", os.path.join(ROOT, "bench_out"))
        self.path = os.path.join(out, f"clocks_gpu{gpu_index}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.f,
                stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                rows.append(parts)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v == "Active"})
        loaded = [v for v in sm if mx and v > 0.3 * max(mx)] or sm
        return dict(sm_mhz=float(np.median(loaded)) if loaded else None,
                    sm_max_mhz=max(mx) if mx else None, reasons=reasons, samples=len(rows))


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

# traced kinds whose trace work is FLOPs on CUDA cores (not tensor cores):
# their rate is GFLOP/s; their HBM rate comes from head_bytes where known
FLOP_KINDS = (10, 11)


def head_bytes(w, plan):
    """Algorithmic HBM bytes of one heads forward and one heads backward of
    the MLP-head tenants in the plan (None if a query head is in the group):
    forward reads W1, b1, W2, b2 (bf16) and the pooled features (fp32) and
    writes the predictions (fp32); backward reads W2 (bf16), the pooled
    features, the cached pre-activations and the output gradients (fp32)
    and writes dW1, db1, dW2, db2 (fp32)."""
    fwd = bwd = 0
    seg = plan.seg_offsets
    for g, t in enumerate(plan.slot_tenant.tolist()):
        tn = w.tenants[t]
        if tn.head_kind != 0:
            return None
        ns = int(seg[g + 1] - seg[g])
        d, hid, wd = w.backbone.d, tn.d_hidden, tn.width
        wts = hid * d + hid + wd * hid + wd
        fwd += 2 * wts + 4 * ns * (d + wd)
        bwd += 2 * (wd * hid) + 4 * ns * (d + hid + wd) + 4 * wts
    return fwd, bwd


def attention_executed_flops(cu_seqlens, H, hd):
    """FLOPs one attention launch executes on the tensor cores: per sample
    of L tokens and query head, ceil(L / 128) query tiles of 128 rows times
    ceil(L / 64) key tiles of 64, for both products (S = Q K^T, O += P V),
    masked entries included."""
    L = np.diff(np.asarray(cu_seqlens, dtype=np.int64))
    rows = -(-L // 128) * 128
    keys = -(-L // 64) * 64
    return float(4.0 * H * hd * np.sum(rows * keys))


def kernel_breakdown(J, kinds, ms, work, bytes_per_launch=None):
    """Per traced kernel kind: launches, total ms, share of the traced time
    and its rate: TFLOP/s for the tcgen05 kinds, GFLOP/s for the head kinds
    (plus GB/s from bytes_per_launch[kind] where given), GB/s of the traced
    bytes otherwise."""
    per_kernel = {}
    tot_ms = float(ms.sum())
    for k in sorted(set(kinds.tolist())):
        m = kinds == k
        name = J.KERNEL_NAMES.get(k, str(k))
        kms = float(ms[m].sum())
        wk = float(work[m].sum())
        rate = wk / (kms / 1e3) if kms > 0 else 0.0
        row = dict(launches=int(m.sum()), ms=round(kms, 3),
                   share=round(kms / tot_ms, 4) if tot_ms else None)
        if k in J.TENSOR_KERNELS:
            row["tflops"] = round(rate / 1e12, 1)
        elif k in FLOP_KINDS:
            row["gflops"] = round(rate / 1e9, 1)
            b = (bytes_per_launch or {}).get(k)
            if b and kms > 0:
                row["gbs"] = round(b * int(m.sum()) / (kms / 1e3) / 1e9, 1)
                row["bytes_per_launch"] = int(b)
        else:
            row["gbs"] = round(rate / 1e9, 1)
        per_kernel[name] = row
    return per_kernel


def run_train(args):
    """One grouped training step of every tenant's LoRA adapters and head on
    the skewed 64-tenant 2B-class workload (rank-16 adapters on Q/K/V/O):
    the shared forward keeping each block's residual input, the tenants'
    heads, losses and feature gradients, then the adapter backward through
    the frozen backbone (each block recomputed from its saved input).
    Tokens/s of the whole step, device-resident inputs, with the per-kernel
    breakdown and the grouped vs per-tenant isolated speedup."""
    import torch

    import synth
    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    from paper_2607_16074_gb300 import runtime as R

    B.build()
    J.lib()
    dev = torch.device("cuda", 0)
    w = make_bench_workload(args)
    if not w.backbone.lora_rank:
        raise SystemExit(f"--train-lora needs a workload with adapters (zipf2b), not {w.name}")
    bw = synth.make_backbone_weights(w, device=dev)
    hw = synth.make_head_weights(w, device=dev)
    inp = synth.make_inputs(w, device=dev)
    reqs = oracle_requests(w)
    plan = J.jnx_group_plan(w.schemas(), reqs, len(w.tenants), w.max_samples, w.max_tokens)
    backbone = R.DeviceBackbone(w.backbone, bw, n_tenants=len(w.tenants))
    heads = R.DeviceHeads(w.tenants, w.backbone.d, hw, device=dev)
    backbone.prepare_backward()
    step = R.LoraTrainStep(backbone, heads, R.DeviceGroup(plan, device=dev), device=dev)
    preds = torch.zeros_like(inp["targets"])
    stream = torch.cuda.current_stream()
    # every group tenant's optimizer step on its own adapters and head
    opt = R.TenantAdamW(backbone.lora_pairs())
    heads.init_optimizer()
    group_tenants = sorted(set(plan.slot_tenant.tolist()))

    def run(st):
        st.run(inp["vision"], inp["text_ids"], inp["targets"], preds)
        tenants = sorted(set(st.group.plan.slot_tenant.tolist()))
        opt.step(tenants, lr=1e-4, weight_decay=0.01)
        heads.adamw_step(st.group, lr=1e-4, weight_decay=0.01)
    for _ in range(max(args.warmup, 3)):
        run(step)
    for ws in (step.ws_bb, step.ws_h, step.ws_bwd):
        R.check_status(ws)
    torch.cuda.synchronize()
    clocks = ClockSampler(0)
    clocks.start()
    cap = 8192 * max(1, args.steps)
    J.jnx_trace_enable(cap)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        run(step)
    e1.record(stream)
    torch.cuda.synchronize()
    launches = J.jnx_trace_count()
    kinds, ms, work = J.jnx_trace_read(cap)
    J.jnx_trace_disable()
    clk = clocks.stop()
    t_ms = e0.elapsed_time(e1)
    tokens = plan.n_tokens
    per_kernel = kernel_breakdown(J, kinds, ms, work)
    peaks = load_peaks()
    # the dominant kernel kind of the step and its roofline
    shares = {k: float(ms[kinds == k].sum()) for k in set(kinds.tolist())}
    top = max(shares, key=shares.get)
    m = kinds == top
    top_rate = float(work[m].sum()) / (float(ms[m].sum()) / 1e3) / 1e12
    roofline = dict(kernel=J.KERNEL_NAMES.get(top, str(top)), bound="tensor",
                    achieved=round(top_rate, 1), peak=peaks["bf16_sustained"], unit="TFLOP/s",
                    frac=round(top_rate / peaks["bf16_sustained"], 4),
                    share_of_step=round(shares[top] / float(ms.sum()), 4),
                    launches_per_step=int(m.sum()) // max(args.steps, 1),
                    peak_note=f"bf16_tflops_sustained of {peaks['source']} peaks")
    # the backward's four input-gradient GEMMs, told apart by their FLOPs per launch
    gb = kinds == 15
    by_shape = {}
    for fl in sorted(set(work[gb].tolist()), reverse=True):
        mm = gb & (work == fl)
        kms = float(ms[mm].sum())
        by_shape["%.3g TFLOP" % (fl / 1e12)] = dict(
            launches=int(mm.sum()), ms=round(kms, 3),
            tflops=round(fl * int(mm.sum()) / (kms / 1e3) / 1e12, 1))
    roofline["gemm_bwd_by_shape"] = by_shape
    bwd_mask = np.isin(kinds, (15, 16, 18))
    bwd_tf = float(work[bwd_mask].sum()) / (float(ms[bwd_mask].sum()) / 1e3) / 1e12
    step_flops = float(work[np.isin(kinds, J.TENSOR_KERNELS)].sum()) / args.steps
    speed = None
    if not args.no_per_tenant:
        del step
        torch.cuda.empty_cache()
        iso = []
        for t in range(len(w.tenants)):
            sub = w.subset([t])
            p = J.jnx_group_plan(sub.schemas(), oracle_requests(sub), len(w.tenants),
                                 w.max_samples, w.max_tokens)
            if p.n_samples:
                iso.append(R.LoraTrainStep(backbone, heads, R.DeviceGroup(p, device=dev),
                                           device=dev))
        for st in iso:
            run(st)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for st in iso:
            run(st)
        b.record(stream)
        torch.cuda.synchronize()
        t_iso = a.elapsed_time(b)
        speed = dict(per_tenant_ms=round(t_iso, 3), grouped_ms=round(t_ms / args.steps, 3),
                     speedup=round(t_iso / (t_ms / args.steps), 4),
                     per_tenant_tokens_per_s=round(tokens / (t_iso / 1e3), 1))
    return dict(metric="lora_train_tokens_per_s", value=round(tokens * args.steps / (t_ms / 1e3), 1),
                unit="tokens/s", steps=args.steps, ms_per_step=round(t_ms / args.steps, 3),
                higher_is_better=True, dtype="bf16", data="synthetic",
                config=dict(workload=workload_desc(w), tokens=tokens, samples=plan.n_samples,
                            tenants=len(w.tenants), lora_rank=w.backbone.lora_rank,
                            step="forward (saving block inputs) + heads + feature gradient + "
                                 "adapter backward (blocks recomputed) + every group tenant's "
                                 "AdamW step on its adapters and head",
                            group_tenants=len(group_tenants)),
                clocks=clk, gpu_launches=int(launches), roofline=roofline,
                backward_tensor=dict(kernels="gemm_bwd + attention_bwd + lora_bwd",
                                     achieved=round(bwd_tf, 1), unit="TFLOP/s",
                                     frac=round(bwd_tf / peaks["bf16_sustained"], 4)),
                step_tensor=dict(achieved=round(step_flops / (t_ms / args.steps / 1e3) / 1e12, 1),
                                 unit="TFLOP/s"),
                per_tenant=speed, kernels=per_kernel)


def run_ours(args, rank, world, local_rank):
    import torch

    import synth
    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    from paper_2607_16074_gb300 import runtime as R

    B.build()
    J.lib()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = make_bench_workload(args)
    # each rank owns an independent group (same shapes, its own inputs)
    w.seed = replica_seed(w.seed, rank)
    bw = synth.make_backbone_weights(w, device=dev)
    hw = synth.make_head_weights(w, device=dev)
    inp = synth.make_inputs(w, device=dev)
    inp_host = {k: v.cpu().pin_memory() for k, v in inp.items()}

    reqs = oracle_requests(w)
    t0 = time.perf_counter()
    plan = J.jnx_group_plan(w.schemas(), reqs, len(w.tenants), w.max_samples, w.max_tokens)
    plan_ms = (time.perf_counter() - t0) * 1e3
    group = R.DeviceGroup(plan, device=dev)
    backbone = R.DeviceBackbone(w.backbone, bw, n_tenants=len(w.tenants))
    heads = R.DeviceHeads(w.tenants, w.backbone.d, hw, device=dev)
    step = R.GroupedStep(backbone, heads, group, device=dev)
    preds = torch.zeros_like(inp["targets"])
    stream = torch.cuda.current_stream()

    def one_step():
        step.run(inp["vision"], inp["text_ids"], inp["targets"], preds)

    for _ in range(args.warmup):
        one_step()
    R.check_status(step.ws_bb)
    R.check_status(step.ws_h)
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    # ---- device-resident timed region, every launch traced ----------------
    clocks = ClockSampler(local_rank)
    clocks.start()
    cap = 4096 * max(1, args.steps)
    barrier()
    torch.cuda.synchronize()
    J.jnx_trace_enable(cap)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        one_step()
    e1.record(stream)
    torch.cuda.synchronize()
    barrier()
    launches = J.jnx_trace_count()
    kinds, ms, work = J.jnx_trace_read(cap)
    J.jnx_trace_disable()
    clk = clocks.stop()
    t_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    tokens = plan.n_tokens
    value = job_tokens_per_s(tokens, world, args.steps, t_ms)

    # ---- end to end through the C ABI from pinned host memory --------------
    # Every step plans its group on the host, copies its inputs from pinned
    # host memory and reads its loss and predictions back; StepPipeline
    # overlaps step i+1's planning and input copy with step i.
    h2d = sum(t.numel() * t.element_size() for t in inp_host.values())
    d2h = step.loss.numel() * 4 + preds.numel() * 4
    pipe = R.StepPipeline(step, inp["vision"].shape[0], inp["text_ids"].numel(),
                          tuple(inp["targets"].shape), device=dev)
    plan_fn = lambda i: J.jnx_group_plan(w.schemas(), reqs, len(w.tenants), w.max_samples,
                                         w.max_tokens)
    pipe.run([inp_host] * 2, plan_fn)  # warm-up of the pipeline's own buffers
    barrier()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    pipe.run([inp_host] * args.steps, plan_fn)
    torch.cuda.synchronize()
    barrier()
    e2e_ms = max_over_ranks((time.perf_counter() - t0) * 1e3, world, dev)
    step.group = group
    e2e_plan_bytes = sum(a.nbytes for a in (plan.cu_seqlens, plan.sample_slot, plan.sample_target,
                                            plan.seg_offsets, plan.gather_src, plan.pos_ids))
    # each step's group also uploads its attention work list
    e2e_plan_bytes += group.d["attn_items"].numel() * 4

    # ---- per-tenant isolated execution (the speedup's baseline) -----------
    speed = None
    if not args.no_per_tenant:
        iso = []
        for t in range(len(w.tenants)):
            sub = w.subset([t])
            p = J.jnx_group_plan(sub.schemas(), oracle_requests(sub), len(w.tenants),
                                 w.max_samples, w.max_tokens)
            if p.n_samples == 0:
                continue
            iso.append(R.GroupedStep(backbone, heads, R.DeviceGroup(p, device=dev), device=dev))
        for st in iso:  # warm
            st.run(inp["vision"], inp["text_ids"], inp["targets"], preds)
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for st in iso:
            st.run(inp["vision"], inp["text_ids"], inp["targets"], preds)
        b.record(stream)
        torch.cuda.synchronize()
        t_iso = a.elapsed_time(b)
        speed = dict(per_tenant_ms=round(t_iso, 3), grouped_ms=round(t_ms / args.steps, 3),
                     speedup=round(t_iso / (t_ms / args.steps), 4),
                     per_tenant_tokens_per_s=round(tokens / (t_iso / 1e3), 1))
        del iso

    # ---- CUDA-graph replay (--graphs): the same steps captured once ---------
    graphs = None
    if args.graphs:
        graphs = graph_timings(args, step, inp, preds, plan, backbone, heads, w, dev, stream)

    # ---- roofline of the dominant kernel (all backbone GEMM launches) ------
    peaks = load_peaks()
    gemm_mask = np.isin(kinds, (3, 5, 6, 7))
    g_flops, g_ms = float(work[gemm_mask].sum()), float(ms[gemm_mask].sum())
    g_tf = g_flops / (g_ms / 1e3) / 1e12 if g_ms > 0 else 0.0
    hb = head_bytes(w, plan)
    per_kernel = kernel_breakdown(J, kinds, ms, work, {10: hb[0], 11: hb[1]} if hb else None)
    att = kinds == 4
    if att.any() and "attention" in per_kernel:
        # the attention row's rate counts 4 L^2 H hd per sample; the kernel
        # also computes the masked parts of its 128-query and 64-key tiles
        ex = attention_executed_flops(plan.cu_seqlens, w.backbone.n_heads, w.backbone.head_dim)
        a_ms = float(ms[att].sum())
        per_kernel["attention"]["tflops_executed"] = round(
            ex * int(att.sum()) / (a_ms / 1e3) / 1e12, 1)
    step_flops = float(work[np.isin(kinds, J.TENSOR_KERNELS + (10, 11))].sum()) / args.steps
    step_tf = step_flops / (t_ms / args.steps / 1e3) / 1e12
    # the dominant kernel: the gate/up projection GEMM (largest share of the step)
    gu = kinds == 6
    gu_n = int(gu.sum())
    gu_flops, gu_ms = float(work[gu].sum()), float(ms[gu].sum())
    gu_tf = gu_flops / (gu_ms / 1e3) / 1e12 if gu_ms > 0 else 0.0
    tr = recorded_traffic(w.name, (plan.n_tokens, w.backbone.d, w.backbone.d_ff))
    roofline = dict(kernel="k_gemm<EPI_GLU> (tcgen05): gate/up projection + SwiGLU/GeGLU",
                    bound="tensor", achieved=round(gu_tf, 1), peak=peaks["bf16_sustained"],
                    unit="TFLOP/s", frac=round(gu_tf / peaks["bf16_sustained"], 4),
                    frac_of_burst=round(gu_tf / peaks["bf16"], 4),
                    share_of_step=round(gu_ms / float(ms.sum()), 4) if gu_n else None,
                    flops_per_launch=gu_flops / max(gu_n, 1),
                    launch_ms=round(gu_ms / max(gu_n, 1), 4),
                    peak_note=f"bf16_tflops_sustained of {peaks['source']} peaks "
                              "(kernel timed inside a long step)",
                    traffic=tr["bytes_per_launch"] if tr else None,
                    algorithmic_bytes_per_launch=gu_algorithmic_bytes(w, plan.n_tokens),
                    traffic_source=tr["source"] if tr else
                    "none recorded for this kernel source and launch shape")
    roofline_all_gemm = dict(kernels="all backbone GEMM launches (QKV+RoPE, O+residual, "
                                     "gate/up+GLU, down+residual)",
                             achieved=round(g_tf, 1), unit="TFLOP/s",
                             frac=round(g_tf / peaks["bf16_sustained"], 4),
                             frac_of_burst=round(g_tf / peaks["bf16"], 4))

    # ---- CPU oracle baseline (rank 0, N = 1 only) --------------------------
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        nl = min(args.oracle_layers, w.backbone.n_layers)
        subset = oracle_tenant_subset(w)
        bw_np, hw_np, inp_np = host_numpy_inputs(w, bw, hw, inp, nl)
        r = oracle_tenant_run(w, subset, nl, bw_np, hw_np, inp_np)
        full_s = oracle_full_depth_s(w, r, nl)
        cpu = dict(value=round(r["tokens"] / full_s, 3), unit="tokens/s", cores=os.cpu_count(),
                   kind="oracle",
                   sample=f"whole tenants {subset} ({r['samples']} samples, {r['tokens']} "
                          f"tokens): backbone through {nl} of {w.backbone.n_layers} blocks, "
                          f"scaled by {w.backbone.n_layers / nl:g} to full depth, plus the "
                          f"heads' forward, loss and gradients as timed",
                   timed_tokens=r["tokens"], timed_blocks=nl,
                   scale=round(w.backbone.n_layers / nl, 3),
                   seconds=round(r["backbone_s"] + r["head_s"], 2))

    out = dict(
        metric=METRIC, value=round(value, 1), unit="tokens/s", n_gpus=world, steps=args.steps,
        warmup=args.warmup, ms_per_step=round(t_ms / args.steps, 3), higher_is_better=True,
        scaling="weak", vs_baseline=None, dtype="bf16", data="synthetic",
        config=dict(workload=workload_desc(w), global_batch=tokens * world,
                    seq_len=int(plan.max_seqlen), parallelism=f"replicas{world}",
                    tenants=len(w.tenants), samples=plan.n_samples,
                    l2="inputs larger than L2 (weights 13 GB, activations > 1 GB per step)"),
        clocks=clk,
        e2e=dict(value=round(job_tokens_per_s(tokens, world, args.steps, e2e_ms), 1),
                 unit="tokens/s",
                 h2d_bytes_per_step=int(h2d + e2e_plan_bytes), d2h_bytes_per_step=int(d2h)),
        gpu_launches=int(launches),
        roofline=roofline,
        roofline_all_gemm=roofline_all_gemm,
        step_tensor=dict(achieved=round(step_tf, 1), unit="TFLOP/s",
                         frac_of_burst=round(step_tf / peaks["bf16"], 4),
                         frac_of_sustained=round(step_tf / peaks["bf16_sustained"], 4),
                         note="algorithmic FLOPs of one step (tensor-core GEMMs and attention, plus the heads' FLOPs, under 0.01 %) / step time"),
        per_tenant=speed,
        plan_ms=round(plan_ms, 3),
        kernels=per_kernel,
        cpu_baseline=cpu,
    )
    if graphs is not None:
        out["graphs"] = graphs
    return out


def graph_timings(args, step, inp, preds, plan, backbone, heads, w, dev, stream):
    """The grouped step, and the per-tenant steps back to back, each captured
    once into a CUDA graph and replayed: K replays timed with CUDA events
    (launch overheads gone from both arms), with the grouped replay's
    predictions checked against the eager step's."""
    import torch

    from paper_2607_16074_gb300 import jnx as J
    from paper_2607_16074_gb300 import runtime as R

    def capture(fn):
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            fn()
        torch.cuda.synchronize()
        return g

    def replay_ms(g):
        for _ in range(max(args.warmup, 3)):
            g.replay()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.steps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) / args.steps

    run = lambda st: st.run(inp["vision"], inp["text_ids"], inp["targets"], preds)
    run(step)
    torch.cuda.synchronize()
    want = preds.clone()
    g = capture(lambda: run(step))
    t_g = replay_ms(g)
    same = bool(torch.equal(preds, want))
    out = dict(ms_per_step=round(t_g, 4),
               value=round(plan.n_tokens / (t_g / 1e3), 1), unit="tokens/s",
               replay_equals_eager=same)
    del g
    if not args.no_per_tenant:
        iso = []
        for t in range(len(w.tenants)):
            sub = w.subset([t])
            p = J.jnx_group_plan(sub.schemas(), oracle_requests(sub), len(w.tenants),
                                 w.max_samples, w.max_tokens)
            if p.n_samples:
                iso.append(R.GroupedStep(backbone, heads, R.DeviceGroup(p, device=dev),
                                         device=dev))
        for st in iso:
            run(st)
        torch.cuda.synchronize()
        gi = capture(lambda: [run(st) for st in iso])
        t_i = replay_ms(gi)
        del gi, iso
        out.update(per_tenant_ms=round(t_i, 4), speedup=round(t_i / t_g, 4))
    return out


def run_reference(args, rank, world):
    """The fp64 CPU oracle, as it stands, timed on the host cores.  One step
    is one whole tenant of the timing subset (oracle_tenant_subset; the
    steps cycle through it) through --reference-layers blocks plus its
    head step; value is the tokens of the timed steps over their time scaled
    to the workload's full depth, ms_per_step the measured wall time of a
    step as run."""
    import synth
    w = synth.make_workload(args.workload)
    nl = min(args.reference_layers, w.backbone.n_layers)
    bw = synth.make_backbone_weights(dataclass_layers(w, nl), device="cpu")
    hw = synth.make_head_weights(w, device="cpu")
    inp = synth.make_inputs(w, device="cpu")
    bw_np, hw_np, inp_np = host_numpy_inputs(w, bw, hw, inp, nl)
    subset = oracle_tenant_subset(w)
    for i in range(args.warmup):
        oracle_tenant_run(w, [subset[i % len(subset)]], nl, bw_np, hw_np, inp_np)
    wall = full = 0.0
    toks = samples = 0
    for i in range(args.steps):
        t0 = time.perf_counter()
        r = oracle_tenant_run(w, [subset[i % len(subset)]], nl, bw_np, hw_np, inp_np)
        wall += time.perf_counter() - t0
        full += oracle_full_depth_s(w, r, nl)
        toks += r["tokens"]
        samples += r["samples"]
    v = toks / full
    desc = (f"one whole tenant per step, cycling through tenants {subset}; backbone through "
            f"{nl} of {w.backbone.n_layers} blocks, scaled by {w.backbone.n_layers / nl:g} to "
            f"full depth, plus the head's forward, loss and gradients as timed")
    return dict(metric=METRIC, value=round(v, 3), unit="tokens/s", n_gpus=world,
                steps=args.steps, warmup=args.warmup,
                ms_per_step=round(wall / max(args.steps, 1) * 1e3, 1), higher_is_better=True,
                scaling="weak", vs_baseline=None, dtype="f64", data="synthetic",
                config=dict(workload=workload_desc(w), parallelism="cpu"),
                impl="reference",
                timed=dict(tokens=toks, samples=samples, blocks=nl,
                           scale=round(w.backbone.n_layers / nl, 3),
                           full_depth_ms_per_step=round(full / max(args.steps, 1) * 1e3, 1),
                           note="ms_per_step is the measured wall time of one step as run "
                                "(nl blocks); value is at full depth"),
                cpu_baseline=dict(value=round(v, 3), unit="tokens/s", cores=os.cpu_count(),
                                  kind="oracle", sample=desc),
                e2e=dict(value=round(v, 3), unit="tokens/s", h2d_bytes_per_step=0,
                         d2h_bytes_per_step=0))


def run_kernel(args):
    """One library kernel alone through the stage-level C ABI on the 7B-class
    shapes with `--tokens` packed rows (samples of 272..320 tokens): a small,
    self-contained case for profilers and per-kernel timing."""
    import torch

    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    B.build()
    L = J.lib()
    dev = torch.device("cuda", 0)
    M, d, F, H, hd = args.tokens, 4096, 11008, 32, 128
    g = torch.Generator(device=dev).manual_seed(7)
    rnd = lambda *s, std=1.0: (torch.randn(*s, generator=g, device=dev) * std).to(torch.bfloat16)
    s = torch.cuda.current_stream()
    rng = np.random.default_rng(7)
    lens = []
    while sum(lens) < M:
        lens.append(int(min(rng.integers(272, 321), M - sum(lens))))
    cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)
    pos = torch.cat([torch.arange(l, dtype=torch.int32) for l in lens]).to(dev)
    ws = torch.zeros(L.jnx_op_gemm_workspace_bytes(1024, hd), dtype=torch.uint8, device=dev)
    k = args.kernel
    if k == "gemm_gu":
        A, W = rnd(M, d), rnd(2 * F, d, std=0.02)
        out = torch.empty(M, F, dtype=torch.bfloat16, device=dev)
        call = lambda: L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), M, 2 * F, d, J.JNX_EPI_GLU,
                                     out.data_ptr(), F, None, 0, 0, 0, 0.0, 0, None, 0, s.cuda_stream)
        work, unit = 2.0 * M * 2 * F * d, "TFLOP/s"
    elif k == "gemm_qkv":
        A, W = rnd(M, d), rnd(3 * d, d, std=0.02)
        out = torch.empty(M, 3 * d, dtype=torch.bfloat16, device=dev)
        call = lambda: L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), M, 3 * d, d, J.JNX_EPI_ROPE,
                                     out.data_ptr(), 3 * d, pos.data_ptr(), 1024, 2 * d, hd,
                                     10000.0, 0, ws.data_ptr(), ws.numel(), s.cuda_stream)
        work, unit = 2.0 * M * 3 * d * d, "TFLOP/s"
    elif k in ("gemm_o", "gemm_down"):
        K = d if k == "gemm_o" else F
        A, W = rnd(M, K), rnd(d, K, std=0.02)
        x = torch.zeros(M, d, dtype=torch.float32, device=dev)
        call = lambda: L.jnx_op_gemm(A.data_ptr(), W.data_ptr(), M, d, K, J.JNX_EPI_RESID,
                                     x.data_ptr(), d, None, 0, 0, 0, 0.0, 0, None, 0, s.cuda_stream)
        work, unit = 2.0 * M * d * K, "TFLOP/s"
    elif k == "attention":
        qkv = rnd(M, 3 * d)
        out = torch.empty(M, d, dtype=torch.bfloat16, device=dev)
        call = lambda: L.jnx_op_attention(qkv.data_ptr(), M, H, H, hd, cu.data_ptr(), len(lens),
                                          max(lens), out.data_ptr(), None, s.cuda_stream)
        work, unit = sum(4.0 * l * l * H * hd for l in lens), "TFLOP/s"
    elif k == "attention_mqa":
        # 2B-class shapes: 8 query heads x 256, one KV head, prefixes of 272..832
        Hq, hdq = 8, 256
        lens = []
        while sum(lens) < M:
            lens.append(int(min(rng.integers(272, 833), M - sum(lens))))
        cu = torch.tensor(np.concatenate([[0], np.cumsum(lens)]), dtype=torch.int32, device=dev)
        qkv = rnd(M, (Hq + 2) * hdq)
        out = torch.empty(M, Hq * hdq, dtype=torch.bfloat16, device=dev)
        call = lambda: L.jnx_op_attention(qkv.data_ptr(), M, Hq, 1, hdq, cu.data_ptr(),
                                          len(lens), max(lens), out.data_ptr(), None,
                                          s.cuda_stream)
        work, unit = sum(4.0 * l * l * Hq * hdq for l in lens), "TFLOP/s"
    elif k == "heads_adamw":
        # the 7B-class group's 32 MLP heads (4096 -> 1024 -> 56): one AdamW
        # step over all of them, 30 bytes per parameter element
        import synth
        from paper_2607_16074_gb300 import runtime as R
        w = synth.make_workload("llama7b")
        hw = synth.make_head_weights(w, device=dev)
        heads = R.DeviceHeads(w.tenants, w.backbone.d, hw, device=dev)
        heads.init_optimizer()
        for gr in heads.grads:
            for v in gr.values():
                v.normal_(generator=g)
        plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                                w.max_tokens)
        grp = R.DeviceGroup(plan, device=dev)
        n_el = sum(v.numel() for gr in heads.grads for v in gr.values())
        call = lambda: (heads.adamw_step(grp, lr=1e-4, weight_decay=0.01), 0)[1]
        work, unit = 30.0 * n_el, "GB/s"
    elif k in ("heads_bwd_adamw", "heads_bwd_then_adamw"):
        # the 7B-class group's 32 MLP heads: the heads backward with the
        # AdamW step fused into it, or the backward then the separate step;
        # both rated on the fused step's algorithmic bytes (weights read for
        # the input gradient, features, moments and masters read and written,
        # bf16 parameters written: 26 bytes per parameter element)
        import synth
        from paper_2607_16074_gb300 import runtime as R
        w = synth.make_workload("llama7b")
        hw = synth.make_head_weights(w, device=dev)
        heads = R.DeviceHeads(w.tenants, w.backbone.d, hw, device=dev)
        heads.init_optimizer()
        plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                                w.max_tokens)
        grp = R.DeviceGroup(plan, device=dev)
        pooled = torch.randn(plan.n_samples, w.backbone.d, generator=g, device=dev)
        tg = synth.make_inputs(w, device=dev)["targets"]
        ws = torch.zeros(heads.workspace_bytes(grp), dtype=torch.uint8, device=dev)
        heads.forward(grp, pooled, None, tg, torch.zeros_like(tg),
                      torch.zeros(len(w.tenants), device=dev), ws)
        n_el = sum(v.numel() for gr in heads.grads for v in gr.values())
        hb = head_bytes(w, plan)[1] - 4 * n_el  # the backward's bytes without its stores
        if k == "heads_bwd_adamw":
            call = lambda: (heads.backward_adamw(grp, pooled, None, tg, ws, lr=1e-4), 0)[1]
        else:
            call = lambda: (heads.backward(grp, pooled, None, tg, ws),
                            heads.adamw_step(grp, lr=1e-4), 0)[2]
        work, unit = hb + 26.0 * n_el, "GB/s"
    elif k == "heads_fwd":
        # the 7B-class group's 32 MLP heads forward and loss on random pooled
        # features, rated on its algorithmic bytes (head_bytes)
        import synth
        from paper_2607_16074_gb300 import runtime as R
        w = synth.make_workload("llama7b")
        hw = synth.make_head_weights(w, device=dev)
        heads = R.DeviceHeads(w.tenants, w.backbone.d, hw, device=dev)
        plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                                w.max_tokens)
        grp = R.DeviceGroup(plan, device=dev)
        pooled = torch.randn(plan.n_samples, w.backbone.d, generator=g, device=dev)
        tg = synth.make_inputs(w, device=dev)["targets"]
        ws = torch.zeros(heads.workspace_bytes(grp), dtype=torch.uint8, device=dev)
        preds, lossb = torch.zeros_like(tg), torch.zeros(len(w.tenants), device=dev)
        call = lambda: (heads.forward(grp, pooled, None, tg, preds, lossb, ws), 0)[1]
        work, unit = head_bytes(w, plan)[0], "GB/s"
    elif k == "pack":
        # the packer over whole 7B-class tenants until --tokens rows: bf16
        # rows read, fp32 rows written (6 bytes per element)
        import synth
        from paper_2607_16074_gb300 import runtime as R
        w = synth.make_workload("llama7b")
        tok, keep = 0, []
        for t in range(len(w.tenants)):
            keep.append(t)
            tok += sum(smp.length(w.backbone.vision_tokens) for r in w.requests if r.tenant == t
                       for smp in r.samples)
            if tok >= M:
                break
        ws_ = w.subset(keep)
        plan = J.jnx_group_plan(ws_.schemas(), oracle_requests(ws_), len(w.tenants), 1 << 30,
                                1 << 30)
        grp = R.DeviceGroup(plan, device=dev)
        inp = synth.make_inputs(w, device=dev)
        tab = rnd(w.backbone.vocab, d)
        x = torch.empty(plan.n_tokens, d, dtype=torch.float32, device=dev)
        call = lambda: L.jnx_op_pack(grp.ref, inp["vision"].data_ptr(), inp["vision"].shape[0],
                                     inp["text_ids"].data_ptr(), inp["text_ids"].shape[0],
                                     tab.data_ptr(), w.backbone.vocab, d, x.data_ptr(), None,
                                     s.cuda_stream)
        work, unit = plan.n_tokens * d * 6.0, "GB/s"
    elif k == "rmsnorm":
        x = torch.randn(M, d, generator=g, device=dev)
        gam = rnd(d)
        out = torch.empty(M, d, dtype=torch.bfloat16, device=dev)
        call = lambda: L.jnx_op_rmsnorm(x.data_ptr(), gam.data_ptr(), 1e-6, M, d, out.data_ptr(),
                                        s.cuda_stream)
        work, unit = M * d * 6.0, "GB/s"
    else:
        raise SystemExit(f"unknown kernel {k}")
    for _ in range(args.warmup):
        J.check(call())
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(s)
        J.check(call())
        b.record(s)
        torch.cuda.synchronize()
        times.append(a.elapsed_time(b))
    med = float(np.median(times))
    rate = work / (med / 1e3) / (1e12 if unit == "TFLOP/s" else 1e9)
    return dict(kernel=k, tokens=M, median_ms=round(med, 4), rate=round(rate, 1), unit=unit,
                times_ms=[round(t, 4) for t in times])


# The flow-expert bench's expert: width 1024, 4 blocks, SwiGLU 4096, chunk 16 x 32.
FLOW_EXPERT = dict(d_model=1024, d_ff=4096, n_blocks=4, chunk=16, action_dim=32)


def flow_workload(T: int, b: int):
    """The flow bench's group on the 2B-class backbone: T tenants x b samples
    of one 256-row image + 16..64 text tokens (seed 43); returns the workload
    and the experts' dimensions (jnx_flow_head fields)."""
    import synth
    bb = synth.Backbone(n_layers=18, d=2048, n_heads=8, n_kv_heads=1, head_dim=256, d_ff=16384,
                        glu=synth.GLU_GEGLU)
    fe = FLOW_EXPERT
    dims = dict(n_tenants=T, d_model=fe["d_model"], d_ff=fe["d_ff"], chunk=fe["chunk"],
                action_dim=fe["action_dim"], d_in=bb.d)
    tenants = [synth.Tenant(synth.HEAD_MLP, chunk=fe["chunk"], action_dim=fe["action_dim"],
                            d_hidden=1024, max_images=1) for _ in range(T)]
    rng = np.random.default_rng(43)
    per = [[synth.Sample(1, int(rng.integers(16, 65))) for _ in range(b)] for _ in range(T)]
    return synth.custom_workload(bb, tenants, per, req_batch=b, seed=43,
                                 name=f"flow{T}x{b}"), dims


def run_flow(args):
    """Flow-matching action experts (DiT heads) as the tenants' modules over
    the shared 2B-class backbone (18 blocks, d=2048, 8x256 query heads on
    one KV head, GeGLU 16384): `--flow-tenants` tenants x `--flow-batch`
    samples (one 256-row image + 16..64 text tokens each; the paper's
    forward breakdown uses 8 x 4), each tenant with a DiT expert of width
    1024, 4 blocks, SwiGLU 4096, chunk 16 x 32.  One training step = the
    shared backbone forward + every tenant's expert forward, rectified-flow
    loss, backward and AdamW step; grouped (one plan) vs serial (each tenant
    alone, back to back).  CUDA events, medians; the tracer gives the breakdown."""
    import dataclasses

    import torch

    import synth
    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    from paper_2607_16074_gb300 import runtime as R

    B.build()
    J.lib()
    dev = torch.device("cuda", 0)
    T, b = args.flow_tenants, args.flow_batch
    w, dims = flow_workload(T, b)
    bb = w.backbone
    bw = synth.make_backbone_weights(w, device=dev)
    backbone = R.DeviceBackbone(bb, bw, n_tenants=T)
    fw = synth.make_flow_weights(T, dims["d_model"], dims["d_ff"], FLOW_EXPERT["n_blocks"],
                                 dims["chunk"], dims["action_dim"], bb.d, 43, device=dev)
    experts = R.DeviceFlowHeads(dims, fw)
    opt = R.TenantAdamW(experts.param_pairs())  # each tenant's expert optimizer
    inp = synth.make_inputs(w, device=dev)
    s = torch.cuda.current_stream()

    class Step:
        def __init__(self, wsub):
            plan = J.jnx_group_plan(wsub.schemas(), oracle_requests(wsub), T, 1 << 30, 1 << 30)
            self.plan, self.g = plan, R.DeviceGroup(plan, device=dev)
            self.ws_bb = torch.zeros(backbone.workspace_bytes(plan.n_tokens), dtype=torch.uint8,
                                     device=dev)
            self.ws_f = torch.zeros(experts.workspace_bytes(self.g), dtype=torch.uint8, device=dev)
            self.hidden = torch.zeros((plan.n_tokens, bb.d), dtype=torch.bfloat16, device=dev)
            self.fi = synth.make_flow_inputs(plan.n_samples, dims["chunk"], dims["action_dim"], 44,
                                             device=dev)
            self.vel = torch.zeros_like(self.fi["actions"])
            self.loss = torch.zeros(T, device=dev)
            self.tenants = sorted(set(plan.slot_tenant.tolist()))

        def backbone(self):
            backbone.forward(self.g, inp["vision"], inp["text_ids"], None, self.hidden, self.ws_bb)

        def expert(self):
            experts.forward(self.g, self.hidden, self.fi["actions"], self.fi["noise"],
                            self.fi["tau"], self.vel, self.loss, self.ws_f)
            experts.backward(self.g, self.hidden, self.ws_f)
            opt.step(self.tenants, lr=1e-4, weight_decay=0.01)

    def timed(fns):
        for _ in range(max(args.warmup, 3)):
            for f in fns:
                f()
        ts = []
        for _ in range(args.steps):
            a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s)
            for f in fns:
                f()
            e.record(s)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(e))
        return float(np.median(ts))

    grouped = Step(w)
    t_bb = timed([grouped.backbone])
    t_ex = timed([grouped.expert])
    t_step = timed([grouped.backbone, grouped.expert])
    R.check_status(grouped.ws_bb)
    R.check_status(grouped.ws_f)
    # the expert's kernels in one traced step
    J.jnx_trace_enable(8192)
    grouped.expert()
    torch.cuda.synchronize()
    kinds, ms, work = J.jnx_trace_read(8192)
    J.jnx_trace_disable()
    expert_kernels = kernel_breakdown(J, kinds, ms, work)
    serial = [Step(w.subset([t])) for t in range(T)]
    t_serial = timed([f for st in serial for f in (st.backbone, st.expert)])
    tokens = grouped.plan.n_tokens
    return dict(metric="flow_expert_train_tokens_per_s",
                value=round(tokens / (t_step / 1e3), 1), unit="tokens/s",
                config=dict(workload=f"{T} tenants x {b} samples ({tokens} tokens) on a 2B-class "
                                     "backbone (18 blocks, d=2048, MQA 8x256, GeGLU 16384)",
                            expert="DiT: width 1024, 4 blocks, 16 heads, SwiGLU 4096, chunk 16 x 32"),
                ms=dict(backbone_forward=round(t_bb, 3), expert_forward_backward=round(t_ex, 3),
                        step=round(t_step, 3), serial_step=round(t_serial, 3)),
                backbone_share_of_step=round(t_bb / t_step, 4),
                speedup_vs_serial=round(t_serial / t_step, 4),
                expert_kernels=expert_kernels)


def run_grid(args):
    """Grouped vs serial inference (backbone forward + head forward, no
    targets) on the grid of tenants {2, 4, 6, 8} x local batch {1, 2, 4, 8}
    samples per tenant, the grid of the paper's group-execution study
    (§5.2).  2B-class backbone (18 blocks, d=2048, 8x256 query heads, one KV
    head, GeGLU 16384), MLP heads, each sample one 256-row image plus 16..64
    text tokens.  Grouped: one plan over all tenants' requests (what
    jnx_sched_poll hands over once the batch reaches B = tenants x local
    batch); serial: each tenant's request planned and run alone, back to
    back.  Speedup = serial time / grouped time (CUDA events, medians)."""
    import dataclasses

    import torch

    import synth
    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    from paper_2607_16074_gb300 import runtime as R

    B.build()
    J.lib()
    dev = torch.device("cuda", 0)
    bb = synth.Backbone(n_layers=18, d=2048, n_heads=8, n_kv_heads=1, head_dim=256, d_ff=16384,
                        glu=synth.GLU_GEGLU)
    T_max, b_max = 8, 8
    tenants = [synth.Tenant(synth.HEAD_MLP, chunk=16, action_dim=7, d_hidden=1024, max_images=1)
               for _ in range(T_max)]
    rng = np.random.default_rng(42)
    lens = rng.integers(16, 65, size=(T_max, b_max))

    def workload(T, b):
        per = [[synth.Sample(1, int(lens[t, i])) for i in range(b)] for t in range(T)]
        w = synth.custom_workload(bb, tenants[:T], per, req_batch=b, seed=42, name=f"grid{T}x{b}")
        return dataclasses.replace(w, tenants=tenants)

    wmax = workload(T_max, b_max)
    bw = synth.make_backbone_weights(wmax, device=dev)
    hw = synth.make_head_weights(wmax, device=dev)
    backbone = R.DeviceBackbone(bb, bw, n_tenants=T_max)
    heads = R.DeviceHeads(tenants, bb.d, hw, device=dev)
    s = torch.cuda.current_stream()

    def timed(fns):
        for _ in range(args.warmup):
            for f in fns:
                f()
        ts = []
        for _ in range(args.steps):
            a, e = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(s)
            for f in fns:
                f()
            e.record(s)
            torch.cuda.synchronize()
            ts.append(a.elapsed_time(e))
        return float(np.median(ts))

    def graph_timed(fns):
        # the same launches captured once into a CUDA graph, then replayed
        for f in fns:
            f()
        cs = torch.cuda.Stream()
        cs.wait_stream(s)
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=cs):
            for f in fns:
                f()
        torch.cuda.synchronize()
        t = timed([gr.replay])
        del gr
        return t

    if args.graphs:
        timed_arm = graph_timed
    else:
        timed_arm = timed

    grid = {}
    for T in (2, 4, 6, 8):
        for b in (1, 2, 4, 8):
            w = workload(T, b)
            inp = synth.make_inputs(w, device=dev)
            preds = torch.zeros_like(inp["targets"])
            plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), T_max, w.max_samples,
                                    w.max_tokens)
            g = R.GroupedStep(backbone, heads, R.DeviceGroup(plan, device=dev), device=dev)
            grouped = timed_arm([lambda g=g: g.infer(inp["vision"], inp["text_ids"], preds)])
            serial_steps = []
            for t in range(T):
                sub = w.subset([t])
                p1 = J.jnx_group_plan(sub.schemas(), oracle_requests(sub), T_max, w.max_samples,
                                      w.max_tokens)
                serial_steps.append(R.GroupedStep(backbone, heads, R.DeviceGroup(p1, device=dev),
                                                  device=dev))
            serial = timed_arm([lambda st=st: st.infer(inp["vision"], inp["text_ids"], preds)
                                for st in serial_steps])
            R.check_status(g.ws_bb)
            grid[f"{T}x{b}"] = dict(tenants=T, local_batch=b, tokens=plan.n_tokens,
                                    grouped_ms=round(grouped, 3), serial_ms=round(serial, 3),
                                    speedup=round(serial / grouped, 3),
                                    grouped_tokens_per_s=round(plan.n_tokens / grouped * 1e3, 1))
            del g, serial_steps, inp, preds
            torch.cuda.empty_cache()
    return dict(metric="grouped vs serial inference forward speedup, tenants x local batch",
                unit="x", higher_is_better=True, n_gpus=1, steps=args.steps,
                warmup=args.warmup, data="synthetic", cuda_graphs=bool(args.graphs),
                config={"workload": "2B-class backbone (18 blocks, d=2048, MQA 8x256, GeGLU "
                                    "16384), MLP heads; samples = 1 image (256 rows) + 16..64 "
                                    "text tokens"},
                grid=grid)


def dataclass_layers(w, n_layers):
    """The workload with only its first n_layers blocks (weights of the other
    blocks are not needed by a bounded oracle sample)."""
    import dataclasses
    return dataclasses.replace(w, backbone=dataclasses.replace(w.backbone, n_layers=n_layers))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama7b")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-per-tenant", action="store_true")
    ap.add_argument("--oracle-layers", type=int, default=2)
    ap.add_argument("--reference-layers", type=int, default=2)
    ap.add_argument("--kernel", default=None,
                    help="time one kernel alone (gemm_gu, gemm_qkv, gemm_o, gemm_down, "
                         "attention, attention_mqa, rmsnorm, heads_adamw, heads_bwd_adamw, "
                         "heads_bwd_then_adamw, pack, heads_fwd) on 7B-class shapes "
                         "with --tokens rows")
    ap.add_argument("--tokens", type=int, default=8192)
    ap.add_argument("--subset", type=int, default=0,
                    help="keep only the first K tenants' requests (a smaller case for profilers)")
    ap.add_argument("--layers", type=int, default=0, help="override the number of blocks")
    ap.add_argument("--grid", default=None, choices=["e4"],
                    help="grouped vs serial inference on the tenants x local batch grid")
    ap.add_argument("--train-lora", action="store_true",
                    help="time the per-tenant LoRA training step (use with --workload zipf2b)")
    ap.add_argument("--graphs", action="store_true",
                    help="also time the grouped and per-tenant steps as CUDA-graph replays")
    ap.add_argument("--flow", action="store_true",
                    help="time flow-matching DiT experts as the tenants' modules")
    ap.add_argument("--flow-tenants", type=int, default=8)
    ap.add_argument("--flow-batch", type=int, default=4)
    args = ap.parse_args()
    if args.flow:
        print(json.dumps(run_flow(args)), flush=True)
        return
    if args.train_lora:
        print(json.dumps(run_train(args)), flush=True)
        return
    if args.grid:
        print(json.dumps(run_grid(args)), flush=True)
        return
    if args.kernel:
        print(json.dumps(run_kernel(args)), flush=True)
        return
    args.warmup = max(args.warmup, 3) if args.impl == "ours" else args.warmup

    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args, rank, world)), flush=True)
        return

    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    out = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
