"""Pins for the oracle's group plan (CPU only)."""
import itertools
import json
import os
import random

import pytest

import synth
from oracle import plan as P
from tests.helpers import oracle_requests

GOLD = os.path.join(os.path.dirname(__file__), "golden", "tiny_plan.json")


def _plan(w, **kw):
    return P.group_plan(w.schemas(), oracle_requests(w), len(w.tenants),
                        kw.get("max_samples", w.max_samples), kw.get("max_tokens", w.max_tokens))


def test_tiny_plan_matches_hand_derived_golden():
    g = json.load(open(GOLD))
    p = _plan(synth.make_workload("tiny"))
    for k in ("n_requests", "n_samples", "n_tokens", "n_slots", "max_seqlen", "cu_seqlens",
              "sample_slot", "sample_req", "sample_target", "sample_width", "seg_offsets",
              "slot_tenant"):
        assert p[k] == g[k], k
    for tok, src in g["gather_spot"].items():
        assert p["gather_src"][int(tok)] == src, tok
    for tok, pos in g["pos_spot"].items():
        assert p["pos_ids"][int(tok)] == pos, tok


def _random_queue(rng, n_req, n_schemas=3, n_tenants=4):
    schemas = []
    for i in range(n_schemas):
        schemas.append(dict(backbone_id=0, d_model=64, vision_tokens=4,
                            embed_dtype=0, vocab_id=100,
                            rope_id=rng.choice([1, 1, 2]),  # some schemas incompatible
                            max_images=2, action_width=rng.choice([3, 5])))
    reqs = []
    vrow = tpos = toff = 0
    for _ in range(n_req):
        t = rng.randrange(n_tenants)
        sc = rng.randrange(n_schemas)
        ss = []
        for _ in range(rng.randint(1, 3)):
            n_img = rng.randint(0, 2)
            tl = rng.randint(0 if n_img else 1, 5)
            ss.append(dict(n_img=n_img, text_len=tl, vision_row=vrow, text_pos=tpos,
                           target_off=toff))
            vrow += n_img * 4
            tpos += tl
            toff += schemas[sc]["action_width"]
        reqs.append(dict(tenant=t, schema=sc, samples=ss))
    return schemas, reqs, n_tenants


def _prefix_valid(schemas, reqs, k, ms, mt):
    """Direct check of one prefix against the acceptance rule."""
    if k == 0:
        return True
    key = P.prefix_signature(schemas[reqs[0]["schema"]])
    if any(P.prefix_signature(schemas[r["schema"]]) != key for r in reqs[:k]):
        return False
    if k == 1:
        return True
    ns = sum(len(r["samples"]) for r in reqs[:k])
    nt = sum(P.sample_length(schemas[r["schema"]], s) for r in reqs[:k] for s in r["samples"])
    return ns <= ms and nt <= mt


def test_prefix_is_the_largest_valid_prefix_brute_force():
    rng = random.Random(7)
    for trial in range(400):
        schemas, reqs, T = _random_queue(rng, rng.randint(0, 5))
        ms, mt = rng.randint(1, 8), rng.randint(1, 40)
        k = P.collect_prefix(schemas, reqs, ms, mt)
        best = max(j for j in range(len(reqs) + 1) if _prefix_valid(schemas, reqs, j, ms, mt)
                   and all(_prefix_valid(schemas, reqs, i, ms, mt) for i in range(j + 1)))
        assert k == best, (trial, k, best)


def test_plan_invariants_random():
    rng = random.Random(11)
    for trial in range(200):
        schemas, reqs, T = _random_queue(rng, rng.randint(1, 6))
        p = P.group_plan(schemas, reqs, T, 1 << 30, 1 << 30)
        acc = reqs[:p["n_requests"]]
        cu = p["cu_seqlens"]
        assert cu[0] == 0 and all(cu[i] < cu[i + 1] for i in range(len(cu) - 1))
        assert cu[-1] == p["n_tokens"] == len(p["gather_src"]) == len(p["pos_ids"])
        # every source row / text position of the accepted samples appears once
        want = []
        for r in acc:
            V = schemas[r["schema"]]["vision_tokens"]
            for s in r["samples"]:
                want += [s["vision_row"] + j for j in range(s["n_img"] * V)]
                want += [-(s["text_pos"] + j) - 1 for j in range(s["text_len"])]
        assert sorted(want) == sorted(p["gather_src"])
        # positions restart at zero in every sample
        for i in range(p["n_samples"]):
            assert p["pos_ids"][cu[i]:cu[i + 1]] == list(range(cu[i + 1] - cu[i]))
        # samples are grouped by slot, slots in order of first appearance
        first = []
        for r in acc:
            if r["tenant"] not in first:
                first.append(r["tenant"])
        assert p["slot_tenant"] == first
        seg = p["seg_offsets"]
        for g in range(p["n_slots"]):
            assert all(p["sample_slot"][i] == g for i in range(seg[g], seg[g + 1]))
            reqs_g = [p["sample_req"][i] for i in range(seg[g], seg[g + 1])]
            assert reqs_g == sorted(reqs_g)  # FIFO within the slot


def test_incompatible_request_stops_the_prefix():
    w = synth.make_workload("tiny")
    sch = w.schemas()
    sch[1]["rope_id"] = 99   # tenant B's schema no longer shares the prefix
    p = P.group_plan(sch, oracle_requests(w), 2, 1 << 30, 1 << 30)
    assert p["n_requests"] == 1 and p["n_slots"] == 1 and p["n_tokens"] == 320


def test_first_request_accepted_even_over_the_limits():
    w = synth.make_workload("tiny")
    p = _plan(w, max_samples=1, max_tokens=1)
    assert p["n_requests"] == 1 and p["n_samples"] == 4


def test_limits_cut_whole_requests():
    w = synth.make_workload("tiny")
    assert _plan(w, max_samples=7)["n_requests"] == 1
    assert _plan(w, max_samples=8)["n_requests"] == 2
    assert _plan(w, max_tokens=671)["n_requests"] == 1
    assert _plan(w, max_tokens=672)["n_requests"] == 2


def test_empty_queue_and_bad_requests():
    w = synth.make_workload("tiny")
    p = P.group_plan(w.schemas(), [], 2, 10, 10)
    assert p["n_samples"] == 0 and p["cu_seqlens"] == [0] and p["n_slots"] == 0
    bad = oracle_requests(w)
    bad[1]["tenant"] = 5
    with pytest.raises(ValueError):
        P.group_plan(w.schemas(), bad, 2, 10, 10)
    bad = oracle_requests(w)
    bad[0]["samples"][0]["n_img"] = 2  # over max_images
    with pytest.raises(ValueError):
        P.group_plan(w.schemas(), bad, 2, 10, 10)
