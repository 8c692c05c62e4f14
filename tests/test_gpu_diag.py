"""Device routines of the hot path on their own, through the C ABI: the
attention softmax's polynomial exponential against 2^x in fp64 over the
whole clamped range, and the bounded wait that every spin in the library's
kernels goes through, made to run out on a barrier nothing arrives on."""
import numpy as np
import pytest
import torch

from paper_2607_16074_gb300 import jnx as J
from tests.gpu_helpers import stream

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2607_16074_gb300 import build as B
    B.build()
    J.lib()


def test_polynomial_exponential_relative_error():
    # a dense grid of [-126, 0] (the softmax's arguments are <= 0 up to the
    # lazy-rescale margin; -126 is the clamp), the integers and half-integers
    # where the range reduction switches, and odd sizes for the pair tail
    x = np.concatenate([np.linspace(-126.0, 0.0, 4_000_001), np.arange(-126, 1) * 1.0,
                        np.arange(-126, 0) + 0.5, [-1e-7, -0.49999997, -0.50000006]])
    x = x.astype(np.float32)
    xd = torch.from_numpy(x).cuda()
    y = torch.full_like(xd, float("nan"))
    J.check(J.lib().jnx_diag_ex2_poly(xd.data_ptr(), y.data_ptr(), x.size, stream()))
    torch.cuda.synchronize()
    ref = np.exp2(x.astype(np.float64))
    got = y.cpu().numpy().astype(np.float64)
    # relative error where the result is a normal number; below x = -125 a
    # result under 2^-126 is subnormal and only its absolute error is bounded
    normal = x >= -125.0
    rel = np.abs(got[normal] / ref[normal] - 1.0)
    ab = np.abs(got[~normal] - ref[~normal])
    print(f"ex2_poly2 over [-125, 0]: max relative error {rel.max():.3e}; "
          f"over [-126, -125): max absolute error {ab.max():.3e}")
    assert rel.max() < 8e-5
    assert ab.max() <= 2.0 ** -125


def test_bounded_wait_gives_up_and_reports_timeout():
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    # a barrier that completes: the wait returns at once, nothing reported
    J.check(J.lib().jnx_diag_bounded_wait(2_000_000, 1, st.data_ptr(), stream()))
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    # nothing ever arrives: the wait gives up after ~1 ms of SM clocks
    J.check(J.lib().jnx_diag_bounded_wait(2_000_000, 0, st.data_ptr(), stream()))
    torch.cuda.synchronize()
    assert int(st.item()) == J.JNX_ERR_TIMEOUT
    # the context is still usable afterwards
    a = torch.ones(1024, device="cuda")
    assert float(a.sum()) == 1024.0
    assert J.lib().jnx_diag_bounded_wait(0, 0, st.data_ptr(), stream()) == J.JNX_ERR_INVALID_ARG
