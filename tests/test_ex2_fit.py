"""The attention softmax's polynomial exponential, pinned on the CPU: the
coefficients compiled into the kernels (jnx_dev.cuh kEx2C0..kEx2C3) are the
minimax (Remez) fit of tests/fit_ex2_poly.py rounded to fp32, the fit
equioscillates as a minimax polynomial must, and its relative error over
[-0.5, 0.5] stays below 8e-5, under the 2^-9 rounding an attention
probability gets when it is stored in bf16."""
import os
import re

import numpy as np

from tests import fit_ex2_poly as F

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                   "paper_2607_16074_gb300", "csrc", "jnx_dev.cuh")


def _compiled():
    s = open(SRC).read()
    return [float(re.search(rf"kEx2C{i} = ([0-9.eE+-]+)f;", s).group(1)) for i in range(4)]


def test_compiled_coefficients_are_the_minimax_fit():
    c, E = F.remez()
    got = np.asarray(_compiled(), dtype=np.float32)
    np.testing.assert_array_equal(got, np.asarray(c, dtype=np.float32))
    assert E < 8e-5


def test_fit_equioscillates_and_bounds_the_error():
    c, E = F.remez()
    xs = np.linspace(F.LO, F.HI, 200001)
    r = np.polyval(np.asarray(c)[::-1], xs) / 2.0 ** xs - 1.0
    # a minimax polynomial of degree 3 touches +-E at 5 alternating points
    sign = np.sign(r)
    runs = np.split(np.arange(xs.size), np.flatnonzero(np.diff(sign) != 0) + 1)
    peaks = [np.max(np.abs(r[run])) for run in runs]
    assert len(peaks) == 5
    assert max(peaks) - min(peaks) < 1e-3 * E
    # the fp32 coefficients keep the bound
    assert F.max_rel_err(np.asarray(_compiled(), dtype=np.float64)) < 8e-5
    # a degree-2 fit could not: the degree is the least that meets 2^-9 / 10
    assert F.remez(degree=2)[1] > 1e-3
