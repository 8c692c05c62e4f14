"""Pins of the flow-matching action-expert oracle (oracle/flow.py): central
finite differences of its loss for every parameter, and closed forms."""
import numpy as np
import pytest

from oracle import flow as Fl
from oracle import model as M

RNG = np.random.default_rng(5)


def _params(dm=8, D=3, C=4, d=6, Fe=10, nb=2, scale=0.4):
    r = lambda *s: scale * RNG.standard_normal(s)
    return dict(w_in=r(dm, D), b_in=r(dm), pos=r(C, dm), t1=r(dm, dm), tb1=r(dm),
                t2=r(dm, dm), tb2=r(dm), w_out=r(D, dm), b_out=r(D),
                blocks=[dict(wqkv=r(3 * dm, dm), wkvc=r(2 * dm, d), wo=r(dm, dm),
                             wg=r(Fe, dm), wu=r(Fe, dm), wd=r(dm, Fe)) for _ in range(nb)])


def _case(n=3, C=4, D=3, d=6):
    ctx = [RNG.standard_normal((L, d)) for L in (1, 5, 9)[:n]]
    acts = RNG.uniform(-1, 1, (n, C, D))
    noise = RNG.standard_normal((n, C, D))
    taus = RNG.uniform(0, 1, n)
    return ctx, acts, noise, taus


def _fd(fn, arr, idx, h=1e-6):
    flat = arr.reshape(-1)
    old = flat[idx]
    flat[idx] = old + h
    lp = fn()
    flat[idx] = old - h
    lm = fn()
    flat[idx] = old
    return (lp - lm) / (2 * h)


def test_gradients_finite_differences_every_parameter():
    p = _params()
    ctx, acts, noise, taus = _case()
    loss, V, g = Fl.tenant_step(p, 2, ctx, acts, noise, taus)
    fn = lambda: Fl.tenant_step(p, 2, ctx, acts, noise, taus)[0]
    pairs = [(p[k], g[k], k) for k in ("w_in", "b_in", "pos", "t1", "tb1", "t2", "tb2",
                                         "w_out", "b_out")]
    for b, (B, G) in enumerate(zip(p["blocks"], g["blocks"])):
        pairs += [(B[k], G[k], (b, k)) for k in B]
    for arr, an, name in pairs:
        assert an.shape == arr.shape, name
        scale = np.abs(an).max()
        for idx in RNG.choice(arr.size, min(arr.size, 6), replace=False):
            fd = _fd(fn, arr, idx)
            assert abs(fd - an.reshape(-1)[idx]) <= 1e-6 * max(abs(fd), scale) + 1e-10, \
                (name, idx, fd, an.reshape(-1)[idx])


def test_identity_blocks_closed_form():
    # W_o = W_d = 0: the blocks add nothing, v = n(h0) W_out^T + b_out
    p = _params()
    for B in p["blocks"]:
        B["wo"][:] = 0
        B["wd"][:] = 0
    X = RNG.standard_normal((5, 6))
    a, e, tau = RNG.uniform(-1, 1, (4, 3)), RNG.standard_normal((4, 3)), 0.3
    x = tau * a + (1 - tau) * e
    s = Fl.time_features(tau, 8)
    phi = p["t2"] @ M.silu(p["t1"] @ s + p["tb1"]) + p["tb2"]
    h0 = x @ p["w_in"].T + p["b_in"] + p["pos"] + phi
    want = h0 / np.sqrt(np.mean(h0 * h0, axis=1, keepdims=True) + 1e-6) @ p["w_out"].T + p["b_out"]
    v, u, _ = Fl.forward(p, 2, X, a, e, tau)
    np.testing.assert_allclose(v, want, rtol=1e-12)
    np.testing.assert_array_equal(u, a - e)


def test_time_features_and_interpolation_ends():
    s = Fl.time_features(0.0, 8)
    np.testing.assert_array_equal(s, [0, 0, 0, 0, 1, 1, 1, 1])
    # tau = 1 feeds the target chunk itself, tau = 0 the noise
    p = _params()
    X = RNG.standard_normal((3, 6))
    a, e = RNG.uniform(-1, 1, (4, 3)), RNG.standard_normal((4, 3))
    np.testing.assert_allclose(Fl.forward(p, 2, X, a, e, 1.0)[0], Fl.network(p, 2, X, a, 1.0)[0],
                               rtol=1e-14)
    np.testing.assert_allclose(Fl.forward(p, 2, X, a, e, 0.0)[0], Fl.network(p, 2, X, e, 0.0)[0],
                               rtol=1e-14)


def test_context_row_order_does_not_matter():
    # attention over the context is a set operation
    p = _params()
    X = RNG.standard_normal((7, 6))
    x = RNG.standard_normal((4, 3))
    v1 = Fl.network(p, 2, X, x, 0.4)[0]
    v2 = Fl.network(p, 2, X[RNG.permutation(7)], x, 0.4)[0]
    np.testing.assert_allclose(v1, v2, rtol=1e-12)
    # ... but the context does matter
    assert not np.allclose(v1, Fl.network(p, 2, X + 1.0, x, 0.4)[0])


def test_zero_loss_zero_gradients_and_constant_velocity_sampling():
    p = _params()
    p["w_out"][:] = 0
    ctx, acts, noise, taus = _case()
    # v = b_out everywhere; targets chosen so that u = a - eps = b_out
    acts = noise + p["b_out"]
    loss, V, g = Fl.tenant_step(p, 2, ctx, acts, noise, taus)
    # zero up to the rounding of (noise + b_out) - noise
    assert loss < 1e-28
    assert all(np.abs(g[k]).max() < 1e-14 for k in g if k != "blocks")
    assert all(np.abs(v).max() < 1e-14 for G in g["blocks"] for v in G.values())
    # Euler integration of a constant velocity is exact
    x1 = Fl.sample(p, 2, ctx[1], noise[1], 7)
    np.testing.assert_allclose(x1, noise[1] + p["b_out"], rtol=1e-13)


def test_norm_backward_finite_differences():
    h = RNG.standard_normal((3, 10))
    dn = RNG.standard_normal((3, 10))
    an = Fl.norm_backward(h, dn)
    fn = lambda: float(np.sum(dn * Fl.norm(h)))
    for idx in range(0, 30, 7):
        fd = _fd(fn, h, idx)
        assert abs(fd - an.reshape(-1)[idx]) < 1e-8
