"""Pins of the AdamW oracle: closed forms, special cases, hand-worked steps
and the library routine torch.optim.AdamW (fp64, CPU)."""
import numpy as np
import pytest
import torch

from oracle import optim as O

HP = dict(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)


def test_first_step_closed_form():
    # at t = 1 the bias corrections give mhat = g and vhat = g^2, so the step
    # is lr * (g / (|g| + eps) + wd * p)
    rng = np.random.default_rng(0)
    p, g = rng.normal(size=50), rng.normal(size=50)
    z = np.zeros(50)
    p1, m1, v1 = O.adamw_step(p, g, z, z, 1, **HP)
    want = p - HP["lr"] * (g / (np.abs(g) + HP["eps"]) + HP["weight_decay"] * p)
    np.testing.assert_allclose(p1, want, rtol=0, atol=1e-15)
    np.testing.assert_allclose(m1, (1 - HP["beta1"]) * g, rtol=1e-15)
    np.testing.assert_allclose(v1, (1 - HP["beta2"]) * g * g, rtol=1e-15)


def test_special_cases():
    rng = np.random.default_rng(1)
    p, g, m, v = (rng.normal(size=20) for _ in range(4))
    v = np.abs(v)
    # lr = 0: the parameter stays, the moments still move
    p1, m1, v1 = O.adamw_step(p, g, m, v, 3, **dict(HP, lr=0.0))
    np.testing.assert_array_equal(p1, p)
    np.testing.assert_allclose(m1, 0.9 * m + 0.1 * g, rtol=1e-15)
    # zero gradient, zero moments, no decay: nothing changes
    z = np.zeros(20)
    p2, m2, v2 = O.adamw_step(p, z, z, z, 1, **dict(HP, weight_decay=0.0))
    np.testing.assert_array_equal(p2, p)
    # zero gradient and moments with decay: pure decoupled decay
    p3, _, _ = O.adamw_step(p, z, z, z, 1, **HP)
    np.testing.assert_allclose(p3, p * (1 - HP["lr"] * HP["weight_decay"]), rtol=1e-15)


def test_two_hand_worked_steps():
    # scalar p = 1, g = 0.5 then g = -0.25, lr = 0.1, beta1 = 0.5, beta2 = 0.75,
    # eps = 0, wd = 0.
    # step 1: m = 0.25, v = 0.0625, mhat = 0.5, vhat = 0.25, p = 1 - 0.1 * 0.5 / 0.5 = 0.9
    # step 2: m = 0.125 - 0.125 = 0, so the update is 0: p stays 0.9;
    #         v = 0.046875 + 0.015625 = 0.0625
    hp = dict(lr=0.1, beta1=0.5, beta2=0.75, eps=0.0, weight_decay=0.0)
    p, m, v = O.adamw_step(1.0, 0.5, 0.0, 0.0, 1, **hp)
    assert float(p) == pytest.approx(0.9, abs=1e-15)
    assert float(m) == 0.25 and float(v) == 0.0625
    p, m, v = O.adamw_step(p, -0.25, m, v, 2, **hp)
    assert float(p) == pytest.approx(0.9, abs=1e-15)
    assert float(m) == 0.0 and float(v) == 0.0625


def test_matches_the_library_adamw_over_several_steps():
    rng = np.random.default_rng(2)
    p0 = rng.normal(size=(7, 5))
    grads = [rng.normal(size=(7, 5)) for _ in range(4)]
    t = torch.tensor(p0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.AdamW([t], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]), eps=HP["eps"],
                            weight_decay=HP["weight_decay"])
    p, m, v = p0, np.zeros_like(p0), np.zeros_like(p0)
    for k, g in enumerate(grads, start=1):
        t.grad = torch.tensor(g, dtype=torch.float64)
        opt.step()
        p, m, v = O.adamw_step(p, g, m, v, k, **HP)
        np.testing.assert_allclose(p, t.detach().numpy(), rtol=1e-13, atol=1e-15)


def test_accumulation_is_the_sum():
    rng = np.random.default_rng(3)
    gs = [rng.normal(size=9) for _ in range(3)]
    np.testing.assert_allclose(O.accumulate(gs), gs[0] + gs[1] + gs[2], rtol=1e-15)
