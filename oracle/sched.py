"""Inference scheduler: when a batch is formed and which queued requests it takes.

Test infrastructure only (see the package docstring).

Paper passages followed:

* §4.3, "Multi-Tenant Group Batching" (its scheduling paragraph): the
  inference service keeps a maximum waiting time T and a target batch size
  B; it takes samples from requests in FIFO order to build a batch and
  starts inference when the waiting time reaches T or the batch size
  reaches B.
* App. A, "Inference Queue Composition": the scheduler looks at the
  requests in arrival order and forms the largest FIFO-compatible prefix the
  batching timeout and maximum batch size allow; compatibility is a property
  of the shared frozen-prefix interface, not of the tenant.

Readings where the paper is silent (each is a choice, not a statement of the paper):

* the waiting time is that of the oldest queued request (now - arrival[0]);
* batch size counts samples, and B is also the batch's sample limit; a
  second limit caps the batch's packed tokens;
* the limits count whole requests; the oldest request is always taken, even
  alone over a limit, so the queue drains;
* compatibility is with the oldest request (equal prefix signatures);
* besides the two triggers, the scheduler also fires when the batch cannot
  grow: the next compatible request in scan order does not fit the limits
  (waiting would only add latency);
* "prefix" mode stops at the first incompatible request (App. A); the
  "skip-ahead" mode passes over incompatible requests (they stay queued, in
  order) and takes later compatible ones, still in arrival order and still
  stopping at the first compatible request that does not fit.
"""
from __future__ import annotations

from typing import Dict, List, Sequence, Tuple

from .plan import prefix_signature, sample_length


def request_tokens(schemas: Sequence[Dict], r: Dict) -> int:
    sc = schemas[r["schema"]]
    return sum(sample_length(sc, s) for s in r["samples"])


def collect(schemas: Sequence[Dict], requests: Sequence[Dict], max_samples: int,
            max_tokens: int, skip_ahead: bool) -> Tuple[List[int], bool]:
    """Indices (ascending) of the requests one batch takes, and whether the
    scan stopped because a compatible request did not fit (batch full)."""
    if not requests:
        return [], False
    head = prefix_signature(schemas[requests[0]["schema"]])
    taken: List[int] = []
    n_s = n_t = 0
    for i, r in enumerate(requests):
        if prefix_signature(schemas[r["schema"]]) != head:
            if skip_ahead:
                continue
            return taken, False
        s, t = len(r["samples"]), request_tokens(schemas, r)
        if taken and (n_s + s > max_samples or n_t + t > max_tokens):
            return taken, True
        taken.append(i)
        n_s += s
        n_t += t
    return taken, False


def poll(schemas: Sequence[Dict], requests: Sequence[Dict], arrival: Sequence[float], now: float,
         timeout: float, batch_samples: int, max_tokens: int,
         skip_ahead: bool) -> Tuple[List[int], float]:
    """(take, wake): the requests to run now (empty: not yet), and, when not
    firing, the time the oldest request's wait reaches the timeout."""
    if not requests:
        return [], float("inf")
    taken, full = collect(schemas, requests, batch_samples, max_tokens, skip_ahead)
    n_s = sum(len(requests[i]["samples"]) for i in taken)
    if n_s >= batch_samples or full or now - arrival[0] >= timeout:
        return taken, now
    return [], arrival[0] + timeout
