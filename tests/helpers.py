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
# Where the CUDA path's own storage formats put the result further than
# BF16_TOL from the fp64 oracle, the GPU may be at most this factor beyond
# the floor those formats alone set (computed in fp64, never on the GPU).
FLOOR_FACTOR = 1.3
# One sample's max|err|/rms is set by a few elements, and at shallow depth
# by where the bf16 output rounding of the GPU and of the emulation happen
# to land; it is gated at this wider factor, the tenant's results as a whole
# at FLOOR_FACTOR.
SAMPLE_FLOOR_FACTOR = 1.5


def gate(floor: float, factor: float = FLOOR_FACTOR) -> float:
    """The bound a floating-point result is held to: the stated BF16_TOL, or
    factor times the floor its storage formats set, if that is larger."""
    return max(BF16_TOL, factor * floor)


def rel_err_bf16_out(got, ref):
    """For outputs stored in bf16: the part of |got - ref| beyond the output
    format's own rounding (half an ulp, at most 2^-8 |ref| for
    round-to-nearest-even), over rms(ref).  A fine-grained check of a
    stage's arithmetic; it never replaces the raw measure (check_bf16_out)."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    if ref.size == 0:
        return 0.0
    rms = float(np.sqrt(np.mean(ref * ref)))
    excess = np.maximum(np.abs(got - ref) - 2.0 ** -8 * np.abs(ref), 0.0)
    return float(np.max(excess)) / max(rms, 1e-300)


def format_floor(ref) -> float:
    """max |bf16(ref) - ref| / rms(ref): how far the exact result itself is
    from its own bf16 rounding, the least error a bf16 output can have."""
    from tests.bf16_emulation import bf16
    return rel_err(bf16(ref), ref)


def check_bf16_out(got, ref, tol_beyond: float, label: str = "", floor=None) -> float:
    """Gate a bf16-stored output on the stated measure, max|err|/rms(ref),
    against gate(floor), and on the part beyond the format's own rounding
    against tol_beyond; prints both.  floor: the error the stage's own
    rounding points set (an emulated result's distance from ref, computed in
    fp64), by default only the output format's (format_floor).  Returns the
    raw measure."""
    raw = rel_err(got, ref)
    fl = format_floor(ref) if floor is None else floor
    beyond = rel_err_bf16_out(got, ref)
    print(f"{label}: max|err|/rms {raw:.3e} (floor {fl:.3e}, gate {gate(fl):.3e}), "
          f"beyond the output rounding {beyond:.3e}")
    assert raw <= gate(fl), (label, "raw", raw, fl)
    assert beyond < tol_beyond, (label, "beyond", beyond, tol_beyond)
    return raw
