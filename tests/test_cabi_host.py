"""CPU tests of the C-ABI library: it loads, exports every symbol the
headers declare, and its host-side plan matches the oracle bit for bit."""
import ctypes as C
import os
import random
import re

import numpy as np
import pytest

import synth
from oracle import plan as OP
from paper_2607_16074_gb300 import build as B
from paper_2607_16074_gb300 import jnx as J
from tests.helpers import oracle_requests
from tests.test_oracle_plan import _random_queue

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module", autouse=True)
def built():
    B.build()


def declared_functions():
    names = set()
    for h in ("jnx.h", "jnx_ops.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(jnx_\w+)\s*\(", src))
    return names


def test_library_exports_every_declared_symbol():
    L = J.lib()
    names = declared_functions()
    assert len(names) >= 16
    for n in names:
        assert hasattr(L, n), n
    assert set(J.EXPORTS) == names
    assert J.jnx_version() == 1


def _cmp(plan, ref):
    for k in J.Plan.FIELDS:
        assert getattr(plan, k).tolist() == ref[k], k
    for k in ("n_requests", "n_samples", "n_tokens", "n_slots", "max_seqlen"):
        assert getattr(plan, k) == ref[k], k


@pytest.mark.parametrize("name", synth.WORKLOADS)
def test_plan_bit_exact_vs_oracle_on_every_workload(name):
    w = synth.make_workload(name)
    reqs = oracle_requests(w)
    for ms, mt in ((1 << 30, 1 << 30), (100, 30000), (3, 1)):
        ref = OP.group_plan(w.schemas(), reqs, len(w.tenants), ms, mt)
        got = J.jnx_group_plan(w.schemas(), reqs, len(w.tenants), ms, mt)
        _cmp(got, ref)


def test_plan_bit_exact_vs_oracle_random_queues():
    rng = random.Random(5)
    for _ in range(300):
        schemas, reqs, T = _random_queue(rng, rng.randint(0, 7))
        ms, mt = rng.randint(1, 9), rng.randint(1, 60)
        _cmp(J.jnx_group_plan(schemas, reqs, T, ms, mt, caps=(1, 1, 1)),
             OP.group_plan(schemas, reqs, T, ms, mt))


def test_plan_errors_write_nothing_and_explain():
    w = synth.make_workload("tiny")
    reqs = oracle_requests(w)
    bad = [dict(r) for r in reqs]
    bad[1] = dict(bad[1], tenant=7)
    with pytest.raises(J.JnxError) as e:
        J.jnx_group_plan(w.schemas(), bad, 2, 100, 1000)
    assert e.value.code == J.JNX_ERR_INVALID_ARG and "tenant" in str(e.value)
    bad = [dict(r) for r in reqs]
    bad[0] = dict(bad[0], samples=[dict(bad[0]["samples"][0], text_len=0, n_img=0)])
    with pytest.raises(J.JnxError):
        J.jnx_group_plan(w.schemas(), bad, 2, 100, 1000)
    bad = [dict(r) for r in reqs]
    bad[0] = dict(bad[0], samples=[dict(bad[0]["samples"][0], vision_row=2**31)])
    with pytest.raises(J.JnxError) as e:
        J.jnx_group_plan(w.schemas(), bad, 2, 100, 1000)
    assert e.value.code == J.JNX_ERR_OVERFLOW


def test_plan_capacity_two_call_pattern():
    w = synth.make_workload("small")
    L = J.lib()
    sch = J.make_schemas(w.schemas())
    req, keep = J.make_requests(oracle_requests(w))
    lim = J.jnx_limits(1 << 30, 1 << 30)
    raw = J.jnx_plan(4, 16, 2, 0, 0, 0, 0, 0, *([None] * 9))
    rc = L.jnx_group_plan(sch, len(w.tenants), req, len(w.requests), len(w.tenants),
                          C.byref(lim), C.byref(raw))
    assert rc == J.JNX_ERR_CAPACITY
    assert raw.n_samples == len(w.samples) and raw.n_tokens == w.n_tokens and raw.n_slots == 8


def test_empty_queue_gives_empty_plan():
    p = J.jnx_group_plan(synth.make_workload("tiny").schemas(), [], 2, 10, 10)
    assert p.n_samples == 0 and p.n_tokens == 0 and p.cu_seqlens.tolist() == [0]


def test_gpu_calls_reject_bad_arguments_without_a_gpu():
    L = J.lib()
    # a null backbone descriptor is rejected on the host before any launch
    rc = L.jnx_backbone_forward(None, None, None, 0, None, 0, None, None, None, 0, None)
    assert rc == J.JNX_ERR_INVALID_ARG
    assert "backbone" in J.jnx_last_error()
    rc = L.jnx_op_gemm(None, None, 1, 256, 64, 0, None, 256, None, 0, 0, 0, 0.0, 0, None, 0, None)
    assert rc == J.JNX_ERR_INVALID_ARG


def _host_group(n_tokens=4):
    """A one-sample, one-slot group whose device arrays are placeholders:
    only its host arrays are read before a call's checks fail."""
    import ctypes as C
    keep = [(C.c_int32 * 2)(0, n_tokens), (C.c_int32 * 2)(0, 1), (C.c_int32 * 1)(0)]
    fake = 1 << 20  # never dereferenced: the calls below return before any launch
    g = J.jnx_group(1, n_tokens, 1, n_tokens, fake, fake, fake, fake, fake, fake,
                    C.cast(keep[0], J.P32), C.cast(keep[1], J.P32), C.cast(keep[2], J.P32))
    return g, keep


def _host_flow_head(d_model):
    import ctypes as C
    fake = 1 << 20
    blocks = (J.jnx_flow_block * 1)(J.jnx_flow_block(fake, fake, fake, fake, fake))
    fh = J.jnx_flow_head(d_model, 256, 1, 8, 7, 256, 1, *([fake] * 9),
                         C.cast(blocks, C.POINTER(J.jnx_flow_block)))
    return fh, blocks


def test_group_attention_work_list():
    """jnx_group_attn_items: every (sample, 128-row tile) of the group once,
    the most expensive first (a sample's cost is its 64-row key tiles), with
    the two-call size query."""
    import ctypes as C
    L = J.lib()
    w = synth.make_workload("small")
    plan = J.jnx_group_plan(w.schemas(), oracle_requests(w), len(w.tenants), w.max_samples,
                            w.max_tokens)
    cu = np.ascontiguousarray(plan.cu_seqlens, dtype=np.int32)
    g = J.jnx_group(plan.n_samples, plan.n_tokens, 0, plan.max_seqlen, *([None] * 6),
                    cu.ctypes.data_as(J.P32), None, None)
    n = L.jnx_group_attn_items(C.byref(g), None, 0)
    lens = np.diff(cu)
    assert n == int(sum((l + 127) // 128 for l in lens))
    out = np.full(2 * n, -1, dtype=np.int32)
    assert L.jnx_group_attn_items(C.byref(g), out.ctypes.data, n - 1) == n  # too small: nothing
    assert (out == -1).all()
    assert L.jnx_group_attn_items(C.byref(g), out.ctypes.data, n) == n
    pairs = out.reshape(n, 2)
    want = sorted((i, t) for i, l in enumerate(lens) for t in range((l + 127) // 128))
    assert sorted(map(tuple, pairs.tolist())) == want
    cost = [(lens[i] + 63) // 64 for i, _ in pairs]
    assert all(a >= b for a, b in zip(cost, cost[1:]))
    assert L.jnx_group_attn_items(None, None, 0) == J.JNX_ERR_INVALID_ARG


def test_training_entry_points_reject_bad_arguments_without_a_gpu():
    import ctypes as C
    L = J.lib()
    inv, uns = J.JNX_ERR_INVALID_ARG, J.JNX_ERR_UNSUPPORTED
    # null descriptors and groups are rejected on the host before any launch
    assert L.jnx_flow_forward(None, None, None, None, None, None, None, None, None, 0, None) == inv
    assert L.jnx_flow_backward(None, None, None, None, 0, None, 0, None) == inv
    assert L.jnx_flow_sample(None, None, None, None, 4, None, None, 0, None) == inv
    assert L.jnx_flow_workspace_bytes(None, None) == 0
    assert L.jnx_backbone_backward_lora(None, None, None, None, None, None, 0, None, 0,
                                        None) == inv
    assert L.jnx_heads_backward_input(None, 0, None, None, None, None, None, None, None, 0,
                                      None) == inv
    assert L.jnx_adamw_tensors(None, 1, None, None) == inv
    assert L.jnx_transpose(None, 1, -1, 4, None, None) == inv
    # a well-formed group: the expert's checks decide, still before any launch
    g, keep = _host_group()
    fh, blocks = _host_flow_head(384)  # width not in {256, 512, 1024}
    fake = 1 << 20
    rc = L.jnx_flow_forward(C.byref(fh), C.byref(g), fake, fake, fake, fake, fake, fake, fake,
                            1 << 30, None)
    assert rc == uns and "d_model" in J.jnx_last_error()
    fh, blocks = _host_flow_head(256)
    rc = L.jnx_flow_forward(C.byref(fh), C.byref(g), fake, fake, fake, fake, fake, fake,
                            fake + 16, 1 << 30, None)  # workspace off a 256-byte boundary
    assert rc == inv and "aligned" in J.jnx_last_error()
    fh.t1 = fake + 2  # a time-MLP weight off a 16-byte boundary
    rc = L.jnx_flow_forward(C.byref(fh), C.byref(g), fake, fake, fake, fake, fake, fake, fake,
                            1 << 30, None)
    assert rc == inv and "aligned" in J.jnx_last_error()


def test_scheduler_bit_exact_vs_oracle_random_queues():
    # jnx_sched_poll (C++) against the scheduler oracle: same queue indices
    # to take and the same wake time, on both collection modes
    from oracle import sched as OS
    from tests.test_oracle_sched import _random_queue as sched_queue
    rng = random.Random(11)
    for _ in range(1500):
        schemas, reqs = sched_queue(rng, rng.randint(0, 8))
        arrival = sorted(rng.uniform(0, 2) for _ in reqs)
        now = (arrival[-1] if arrival else 0.0) + rng.uniform(0, 1.5)
        T, Bs, mt = rng.uniform(0.0, 1.5), rng.randint(1, 12), rng.randint(1, 90)
        skip = rng.random() < 0.5
        want = OS.poll(schemas, reqs, arrival, now, T, Bs, mt, skip)
        got = J.jnx_sched_poll(schemas, reqs, arrival, 4, now, T, Bs, mt, skip)
        assert got == want


def test_scheduler_rejects_bad_policies_and_requests():
    from tests.test_oracle_sched import _random_queue as sched_queue
    schemas, reqs = sched_queue(random.Random(3), 3)
    for kw in (dict(batch_samples=0), dict(max_tokens=0), dict(timeout=-1.0)):
        args = dict(timeout=1.0, batch_samples=4, max_tokens=64)
        args.update(kw)
        with pytest.raises(J.JnxError) as e:
            J.jnx_sched_poll(schemas, reqs, [0.0, 0.1, 0.2], 4, 0.5, **args)
        assert e.value.code == J.JNX_ERR_INVALID_ARG
    bad = [dict(reqs[0], tenant=9)] + reqs[1:]
    with pytest.raises(J.JnxError):
        J.jnx_sched_poll(schemas, bad, [0.0, 0.1, 0.2], 4, 0.5, 1.0, 4, 64)
