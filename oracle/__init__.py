"""fp64 CPU oracle for the grouped multi-tenant path — TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may import this package.  The product path (the CUDA
library and its Python binding) never calls it, and it never calls them: the
two share no code.  Inputs reach both sides from the seeded generators in
``synth``.

What it computes, and where the paper defines it:

* ``plan``   — the FIFO-compatible prefix of inference requests and the
  canonical packed batch with its slices (App. A, "Inference Queue
  Composition": requests examined in arrival order, the largest compatible
  prefix under the batch limits, compatibility decided at the shared
  frozen-prefix boundary; §4.3 "Multi-Tenant Group Batching": the canonical
  VLAFeature is the concatenation point).
* ``model``  — the shared frozen backbone forward, the tenant-private action
  heads, the per-tenant L2 loss and the head gradients.  The grouped method
  must reach exactly what isolated per-tenant execution computes (§5.2: group
  execution concatenates compatible inputs for one shared forward and then
  splits features for tenant-private loss and backward; App. A: nothing is
  averaged across tenants).  So the oracle is that plain definition: every
  sample runs through the backbone on its own, every tenant's head, loss and
  gradient see only that tenant's samples.

The paper prints no layer equations, no head definition and no numeric
result for this path (its §5.2 figures carry no numbers in the text).  The
readings taken where it is silent are listed in the header of ``model``.
Each function is pinned by something other than itself — closed forms,
special cases that reduce to a textbook result, brute force on tiny inputs,
central finite differences for every gradient, and the grouped == isolated
and slot-isolation invariants — and the plan additionally by a hand-derived
example of the tiny workload (``tests/golden``).
"""
