"""Group plan: FIFO-compatible prefix collection and canonical packing.

Test infrastructure only (see the package docstring).

Paper passages followed:

* App. A, "Inference Queue Composition": the Inference Scheduler looks at the
  requests in arrival order and forms the largest FIFO-compatible prefix the
  batch limits allow; compatibility is a property of the shared frozen-prefix
  interface (same base-model interface, same model-specific shape
  constraints), not of tenant identity; canonicalisation then yields one
  physical encoder batch together with the slices that route features back.
* §4.3, "Multi-Tenant Group Batching": the canonical VLAFeature is where
  samples of different tenants are concatenated; features are afterwards
  partitioned to each tenant's action module.

Readings where the paper is silent (each is a choice, not a statement of the paper):

* compatibility = equality of the prefix signature (backbone id, width,
  vision tokens per image, embedding dtype, vocabulary id, RoPE id);
* the scan stops at the first incompatible request (a prefix, no skipping);
* the batch limits count whole requests (samples and tokens); the first
  request is always accepted, even alone over a limit, so the queue drains;
* varlen packing with no padding; position ids restart at 0 in every sample;
* packed order: tenants in order of first appearance, then their requests in
  arrival order, then each request's samples in order; inside a sample the
  vision rows of image 0..k-1 come first, then the text tokens.
"""
from __future__ import annotations

from typing import Dict, List, Sequence

PREFIX_KEYS = ("backbone_id", "d_model", "vision_tokens", "embed_dtype", "vocab_id", "rope_id")


def prefix_signature(schema: Dict) -> tuple:
    """The part of a schema that decides compatibility at the shared prefix."""
    return tuple(int(schema[k]) for k in PREFIX_KEYS)


def validate(schemas: Sequence[Dict], requests: Sequence[Dict], n_tenants: int) -> None:
    """Reject malformed requests (raises ValueError)."""
    for i, r in enumerate(requests):
        if not (0 <= r["tenant"] < n_tenants):
            raise ValueError(f"request {i}: tenant {r['tenant']} outside [0, {n_tenants})")
        if not (0 <= r["schema"] < len(schemas)):
            raise ValueError(f"request {i}: schema {r['schema']} out of range")
        if len(r["samples"]) < 1:
            raise ValueError(f"request {i}: no samples")
        sc = schemas[r["schema"]]
        for s in r["samples"]:
            if not (0 <= s["n_img"] <= sc["max_images"]) or s["text_len"] < 0:
                raise ValueError(f"request {i}: bad sample shape {s}")
            if s["n_img"] * sc["vision_tokens"] + s["text_len"] < 1:
                raise ValueError(f"request {i}: empty sample")


def sample_length(schema: Dict, s: Dict) -> int:
    return s["n_img"] * schema["vision_tokens"] + s["text_len"]


def collect_prefix(schemas, requests, max_samples: int, max_tokens: int) -> int:
    """Number of requests in the largest FIFO-compatible prefix."""
    if not requests:
        return 0
    key = prefix_signature(schemas[requests[0]["schema"]])
    n_samples = n_tokens = 0
    k = 0
    for r in requests:
        sc = schemas[r["schema"]]
        if prefix_signature(sc) != key:
            break
        rs = len(r["samples"])
        rt = sum(sample_length(sc, s) for s in r["samples"])
        if k > 0 and (n_samples + rs > max_samples or n_tokens + rt > max_tokens):
            break
        n_samples += rs
        n_tokens += rt
        k += 1
    return k


def group_plan(schemas: Sequence[Dict], requests: Sequence[Dict], n_tenants: int,
               max_samples: int, max_tokens: int) -> Dict:
    """Collect the prefix and canonicalise it into one packed varlen batch.

    Returns plain Python lists:
      n_requests, n_samples, n_tokens, n_slots, max_seqlen
      cu_seqlens[S+1]   token offset of each packed sample
      sample_slot[S]    group slot (0..n_slots-1) of each packed sample
      sample_req[S]     accepted request index of each packed sample
      sample_target[S]  offset of the sample's targets / predictions
      sample_width[S]   number of action outputs of the sample (C * D_t)
      seg_offsets[G+1]  packed-sample offset of each group slot
      slot_tenant[G]    tenant slot of each group slot
      gather_src[N]     per token: vision row (>= 0) or -(text position + 1)
      pos_ids[N]        per token position inside its sample
    """
    validate(schemas, requests, n_tenants)
    k = collect_prefix(schemas, requests, max_samples, max_tokens)
    acc = list(requests[:k])

    slot_tenant: List[int] = []
    for r in acc:
        if r["tenant"] not in slot_tenant:
            slot_tenant.append(r["tenant"])

    cu, sslot, sreq, stgt, swid, seg = [0], [], [], [], [], [0]
    gather, pos = [], []
    for g, t in enumerate(slot_tenant):
        for ri, r in enumerate(acc):
            if r["tenant"] != t:
                continue
            sc = schemas[r["schema"]]
            V = sc["vision_tokens"]
            for s in r["samples"]:
                L = sample_length(sc, s)
                for j in range(s["n_img"] * V):
                    gather.append(s["vision_row"] + j)
                for j in range(s["text_len"]):
                    gather.append(-(s["text_pos"] + j) - 1)
                pos.extend(range(L))
                cu.append(cu[-1] + L)
                sslot.append(g)
                sreq.append(ri)
                stgt.append(s["target_off"])
                swid.append(sc["action_width"])
        seg.append(len(sslot))

    S = len(sslot)
    return dict(n_requests=k, n_samples=S, n_tokens=cu[-1], n_slots=len(slot_tenant),
                max_seqlen=max((cu[i + 1] - cu[i] for i in range(S)), default=0),
                cu_seqlens=cu, sample_slot=sslot, sample_req=sreq, sample_target=stgt,
                sample_width=swid, seg_offsets=seg, slot_tenant=slot_tenant,
                gather_src=gather, pos_ids=pos)
