"""Shared test helpers: convert synth workloads into the plain structures
the oracle and the C-ABI take, and the parity measure used throughout."""
import numpy as np


def oracle_requests(w):
    return [dict(tenant=r.tenant, schema=r.schema,
                 samples=[dict(n_img=s.n_img, text_len=s.text_len, vision_row=s.vision_row,
                               text_pos=s.text_pos, target_off=s.target_off)
                          for s in r.samples])
            for r in w.requests]


def rel_err(got, ref):
    """max |got - ref| / rms(ref): the parity measure for floating point."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    rms = float(np.sqrt(np.mean(ref * ref))) if ref.size else 0.0
    if ref.size == 0:
        return 0.0
    return float(np.max(np.abs(got - ref))) / max(rms, 1e-300)


BF16_TOL = 2e-2      # GPU (bf16 storage, fp32 accumulation) vs the fp64 oracle
GROUPED_TOL = 1e-3   # GPU grouped vs GPU per-tenant isolated


def deep_tol(n_layers: int) -> float:
    """Bound for whole-path features after n_layers bf16 blocks.

    The tensor-core GEMMs read their inputs (the normed activations and the
    FFN intermediate) in bf16, so every block adds independent relative noise
    of order 2^-9 and the error grows as sqrt(L).  On the 7B-class shapes an
    fp64 emulation of exactly these rounding points lands at about
    0.0105 * sqrt(L) of rms on one sample's pooled feature (0.011 at L=1,
    0.021 at 4, 0.040 at 16, 0.057 at 32).  The bound is the stated 2e-2 per
    block, scaled by sqrt(L): 2e-2 * sqrt(L)."""
    return BF16_TOL * max(1, n_layers) ** 0.5


def rel_err_bf16_out(got, ref):
    """Parity measure for outputs stored in bf16: the part of |got - ref|
    beyond the output format's own rounding (half an ulp, at most 2^-8 |ref|
    for round-to-nearest-even), over rms(ref)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if ref.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(ref * ref)))
    excess = np.maximum(np.abs(got - ref) - 2.0 ** -8 * np.abs(ref), 0.0)
    return float(np.max(excess)) / max(rms, 1e-300)


def grad_tols(head_kind, hw, feats, targets, feat_tol, trials=5, seed=0):
    """Bound for whole-path head gradients given the bound on the features.

    The head stage itself is checked to 1e-4 on synthetic features, so a
    gradient's whole-path error is the backbone's feature error carried
    through the head.  Head gradients are sums of outer products (dW1 =
    dz^T p), and max|err|/rms multiplies the peak-to-rms ratios of both
    factors, so the same feature error shows up larger there.  This measures
    that amplification on the oracle alone: random feature perturbations
    whose max equals feat_tol x rms(features) are pushed through the oracle's
    head step, and each gradient's bound is 2x the largest shift seen
    (never below feat_tol)."""
    from oracle import model as M
    rng = np.random.default_rng(seed)
    base = M.tenant_step(head_kind, hw, feats, targets)[2]
    allf = np.concatenate([np.ravel(f) for f in feats])
    rms = float(np.sqrt(np.mean(allf * allf)))
    worst = {k: 0.0 for k in base}
    for _ in range(trials):
        pert = []
        for f in feats:
            n = rng.standard_normal(np.shape(f))
            pert.append(np.asarray(f) + n / np.max(np.abs(n)) * feat_tol * rms)
        g = M.tenant_step(head_kind, hw, pert, targets)[2]
        for k in base:
            worst[k] = max(worst[k], rel_err(g[k], base[k]))
    return {k: max(feat_tol, 2.0 * v) for k, v in worst.items()}
