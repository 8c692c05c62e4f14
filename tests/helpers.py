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
