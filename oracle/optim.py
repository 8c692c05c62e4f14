"""Tenant-private optimizer step for the heads: AdamW with decoupled weight decay.

Test infrastructure only (see the package docstring).

Paper passages followed:

* App. A, "Actor Consumption and Version Consistency": an optimizer
  microbatch holds one tenant-schema group; the actor activates that
  tenant's action module and optimizer, computes its loss, runs backward and
  the optimizer step, and increments only that tenant's policy version;
  losses, gradients, optimizer states and version counters are never
  averaged across tenants.
* §4.2, "Server Backend" (its Training Queue paragraph): training activates
  the action module and optimizer state of the job's tenant.

Readings where the paper is silent (each is a choice, not a statement of the paper):

* the optimizer is AdamW (Adam moments with bias correction; weight decay
  decoupled from the gradient and applied to the parameter before the step);
  its hyperparameters (lr, beta1, beta2, eps, weight_decay) come from the
  caller, and the step counter t counts steps already taken plus this one;
* updates act on an fp32 master copy of each head parameter; the bf16
  parameter the forward reads is the master rounded to nearest even;
* a tenant's policy version counts its optimizer steps;
* gradient accumulation sums the gradients of successive backward calls.

The update of one parameter element, with g its gradient:

    m <- beta1 m + (1 - beta1) g
    v <- beta2 v + (1 - beta2) g^2
    p <- p - lr * ( (m / (1 - beta1^t)) / (sqrt(v / (1 - beta2^t)) + eps)
                    + weight_decay * p )
"""
from __future__ import annotations

import numpy as np


def adamw_step(p, g, m, v, t: int, lr: float, beta1: float, beta2: float, eps: float,
               weight_decay: float):
    """One AdamW step in fp64 on arrays (returns new p, m, v).  t >= 1 is the
    number of this step."""
    p, g, m, v = (np.asarray(a, dtype=np.float64) for a in (p, g, m, v))
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    mhat = m / (1.0 - beta1 ** t)
    vhat = v / (1.0 - beta2 ** t)
    p = p - lr * (mhat / (np.sqrt(vhat) + eps) + weight_decay * p)
    return p, m, v


def accumulate(grads):
    """Gradient accumulation over successive backward calls: their sum."""
    out = None
    for g in grads:
        g = np.asarray(g, dtype=np.float64)
        out = g.copy() if out is None else out + g
    return out
