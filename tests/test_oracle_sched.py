"""Pins of the inference-scheduler oracle (trigger and collection), against
hand-worked cases and against the definitions restated by enumeration."""
import json
import os
import random

import pytest

from oracle import sched as S
from oracle.plan import prefix_signature

HERE = os.path.dirname(__file__)


def _golden():
    with open(os.path.join(HERE, "golden", "sched_cases.json")) as f:
        return json.load(f)


def _req(spec):
    return {"tenant": spec["tenant"], "schema": spec["schema"],
            "samples": [{"n_img": a, "text_len": b} for a, b in spec["samples"]]}


@pytest.mark.parametrize("case", _golden()["cases"], ids=lambda c: c["name"][:40])
def test_hand_worked_cases(case):
    g = _golden()
    reqs = [_req(g["requests"][k]) for k in case["queue"]]
    take, wake = S.poll(g["schemas"], reqs, case["arrival"], case["now"], case["T"], case["B"],
                        case["max_tokens"], case["skip_ahead"])
    assert take == case["take"]
    assert wake == (float("inf") if case["wake"] is None else case["wake"])


def _random_queue(rng, n):
    schemas = [
        {"backbone_id": 1, "d_model": 64, "vision_tokens": 4, "embed_dtype": 0, "vocab_id": 0,
         "rope_id": 0, "max_images": 3, "action_width": 7},
        {"backbone_id": 1, "d_model": 64, "vision_tokens": 4, "embed_dtype": 0, "vocab_id": 0,
         "rope_id": 0, "max_images": 3, "action_width": 14},
        {"backbone_id": 2, "d_model": 64, "vision_tokens": 4, "embed_dtype": 0, "vocab_id": 0,
         "rope_id": 0, "max_images": 3, "action_width": 7},
    ]
    reqs = []
    for _ in range(n):
        k = rng.randint(1, 4)
        reqs.append({"tenant": rng.randint(0, 3), "schema": rng.randint(0, 2),
                     "samples": [{"n_img": rng.randint(0, 2), "text_len": rng.randint(1, 9)}
                                 for _ in range(k)]})
    return schemas, reqs


def _fits(schemas, reqs, idx, max_s, max_t):
    return (sum(len(reqs[i]["samples"]) for i in idx) <= max_s
            and sum(S.request_tokens(schemas, reqs[i]) for i in idx) <= max_t)


def test_prefix_mode_is_the_longest_admissible_prefix():
    # the definition, by enumeration: the longest prefix whose requests all
    # share the oldest request's signature and that fits the limits (a
    # one-request prefix always qualifies)
    rng = random.Random(5)
    for _ in range(3000):
        schemas, reqs = _random_queue(rng, rng.randint(1, 7))
        max_s, max_t = rng.randint(1, 12), rng.randint(1, 80)
        head = prefix_signature(schemas[reqs[0]["schema"]])
        best = 1
        for k in range(1, len(reqs) + 1):
            idx = list(range(k))
            if all(prefix_signature(schemas[reqs[i]["schema"]]) == head for i in idx) and \
                    (k == 1 or _fits(schemas, reqs, idx, max_s, max_t)):
                best = k
        taken, _ = S.collect(schemas, reqs, max_s, max_t, skip_ahead=False)
        assert taken == list(range(best))


def test_skip_ahead_is_the_longest_admissible_prefix_of_the_compatible_requests():
    rng = random.Random(6)
    for _ in range(3000):
        schemas, reqs = _random_queue(rng, rng.randint(1, 7))
        max_s, max_t = rng.randint(1, 12), rng.randint(1, 80)
        head = prefix_signature(schemas[reqs[0]["schema"]])
        comp = [i for i, r in enumerate(reqs) if prefix_signature(schemas[r["schema"]]) == head]
        best = 1
        for k in range(1, len(comp) + 1):
            if k == 1 or _fits(schemas, reqs, comp[:k], max_s, max_t):
                best = k
        taken, _ = S.collect(schemas, reqs, max_s, max_t, skip_ahead=True)
        assert taken == comp[:best]
        # the prefix mode's batch is always the start of the skip-ahead batch
        pre, _ = S.collect(schemas, reqs, max_s, max_t, skip_ahead=False)
        assert taken[:len(pre)] == pre


def test_trigger_fires_exactly_on_b_full_or_timeout():
    rng = random.Random(7)
    for _ in range(2000):
        schemas, reqs = _random_queue(rng, rng.randint(1, 6))
        arrival = sorted(rng.uniform(0, 1) for _ in reqs)
        T, B, max_t = rng.uniform(0.1, 1.0), rng.randint(1, 10), rng.randint(5, 80)
        now = arrival[-1] + rng.uniform(0, 1.2)
        skip = rng.random() < 0.5
        take, wake = S.poll(schemas, reqs, arrival, now, T, B, max_t, skip)
        coll, _ = S.collect(schemas, reqs, B, max_t, skip)
        n_s = sum(len(reqs[i]["samples"]) for i in coll)
        # "full": the next compatible request after the batch exists and does not fit
        head = prefix_signature(schemas[reqs[0]["schema"]])
        after = [i for i in range(len(reqs)) if i > coll[-1]
                 and prefix_signature(schemas[reqs[i]["schema"]]) == head]
        nxt = after[0] if after else None
        if nxt is not None and not skip:
            # in prefix mode the next request must directly follow the batch
            nxt = nxt if nxt == coll[-1] + 1 else None
        full = nxt is not None and not _fits(schemas, reqs, coll + [nxt], B, max_t)
        should = n_s >= B or full or now - arrival[0] >= T
        assert (take == coll) if should else (take == [] and wake == arrival[0] + T)
