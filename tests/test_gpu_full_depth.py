"""Full-depth parity of the grouped path against the oracle, measured in the
stated measure (max |err| / rms(ref), nothing subtracted) and gated against
the floor that the CUDA path's own storage formats set.

The CUDA path reads every GEMM operand in bf16 and keeps its residual
stream in fp32, so after 18 or 32 blocks its features cannot match the fp64
oracle to 2e-2 of rms: those roundings alone, applied in fp64 at exactly
the kernels' rounding points (tests/bf16_emulation.py, pinned on the CPU),
land near 0.05 on the 7B-class shapes.  Each test here runs the workload's
full group on the GPU at full depth in the benchmark's launch configuration,
then computes, for whole tenants, the oracle's per-sample forward and the
emulated forward on the same inputs, and asserts, per sample and per head
quantity, that the GPU's error is within max(2e-2, 1.3 x the emulated
floor) (tests/helpers.py gate).  Every number is printed (pytest -s).

Paper passages: §5.2 (one shared backbone pass gives every tenant what its
own pass would), App. A "Actor Consumption and Version Consistency"
(tenant-private loss and head gradients)."""
import pytest

import synth
from tests.gpu_helpers import Setup, check_tenants, tenant_samples

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    from paper_2607_16074_gb300 import jnx as J
    B.build()
    J.lib()


def _check(name, s, plan, step, preds, pick):
    # every quantity is gated inside check_tenants; at full depth the
    # features' floors exceed BF16_TOL / FLOOR_FACTOR, so their gate is
    # FLOOR_FACTOR times the floor
    check_tenants(name, s, plan, step, preds, pick)


def test_llama7b_full_depth_two_smallest_tenants():
    """32 blocks, d = 4096, the whole 65,817-token group (the benchmark's
    launch configuration); every sample of the two tenants with the fewest
    samples (6 each) checked end to end: pooled features, predictions, loss
    and head gradients."""
    w = synth.make_workload("llama7b")
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    counts = {t: len(tenant_samples(w, t)) for t in range(len(w.tenants))}
    pick = sorted(counts, key=lambda t: (counts[t], t))[:2]
    _check("llama7b", s, plan, step, preds, pick)


def test_mqa2b_full_depth_smallest_tenant():
    """18 blocks of the 2B-class MQA backbone (8 x 256 query heads, one K/V
    head, GeGLU 16384) over the whole 16-tenant group; the tenant with the
    fewest tokens (16 samples) checked end to end through its query head:
    final normed rows of every sample, predictions, loss, head gradients."""
    w = synth.make_workload("mqa2b")
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    tok = {t: sum(smp.length(w.backbone.vision_tokens) for smp in tenant_samples(w, t))
           for t in range(len(w.tenants))}
    pick = [min(tok, key=lambda t: (tok[t], t))]
    _check("mqa2b", s, plan, step, preds, pick)


def test_zipf2b_full_depth_one_tenant_with_adapters():
    """18 blocks of the skewed 64-tenant group with per-tenant LoRA (rank 16
    on Q/K/V/O); the tenant with the fewest tokens among those with at least
    four samples checked end to end through its adapters and query head."""
    w = synth.make_workload("zipf2b")
    s = Setup(w, gen_device="cuda")
    plan, step, preds = s.run()
    v = w.backbone.vision_tokens
    tok = {t: sum(smp.length(v) for smp in tenant_samples(w, t))
           for t in range(len(w.tenants)) if len(tenant_samples(w, t)) >= 4}
    pick = [min(tok, key=lambda t: (tok[t], t))]
    _check("zipf2b", s, plan, step, preds, pick)
