"""Minimax fit of the degree-3 polynomial that the varlen attention's
softmax uses for 2^f on f in [-0.5, 0.5] (one exponential in four is taken
off the MUFU pipe this way: 2^x = 2^j 2^f with j = rint(x)).

Method: the Remez exchange algorithm for the relative error
r(f) = p(f) / 2^f - 1.  Start from Chebyshev extrema as the reference
points, solve the linear system p(f_i) - 2^(f_i) = (-1)^i E 2^(f_i) for the
four coefficients and the levelled error E, move the reference to the
alternating extrema of r on a dense grid, and repeat until E settles.  The
result equioscillates at five points with |r| = |E|.

    python tests/fit_ex2_poly.py      # prints the coefficients and |E|
"""
import numpy as np

DEGREE = 3
LO, HI = -0.5, 0.5


def remez(degree: int = DEGREE, iters: int = 30, grid: int = 200001):
    n = degree + 2
    k = np.arange(n)
    ref = 0.5 * (LO + HI) - 0.5 * (HI - LO) * np.cos(np.pi * k / (n - 1))
    xs = np.linspace(LO, HI, grid)
    E = 0.0
    for _ in range(iters):
        A = np.zeros((n, n))
        for i, x in enumerate(ref):
            A[i, :degree + 1] = x ** np.arange(degree + 1)
            A[i, degree + 1] = -((-1) ** i) * 2.0 ** x
        sol = np.linalg.solve(A, 2.0 ** ref)
        c, E = sol[:degree + 1], sol[degree + 1]
        r = np.polyval(c[::-1], xs) / 2.0 ** xs - 1.0
        # one extremum per run of constant sign, ends included
        sign = np.sign(r)
        cut = np.flatnonzero(np.diff(sign) != 0) + 1
        runs = np.split(np.arange(grid), cut)
        ext = [run[np.argmax(np.abs(r[run]))] for run in runs if len(run)]
        if len(ext) < n:
            break
        # keep n alternating extrema with the largest magnitudes in order
        while len(ext) > n:
            i = int(np.argmin([abs(r[e]) for e in ext]))
            ext.pop(i)
        new = xs[ext]
        if np.allclose(new, ref, atol=1e-12):
            break
        ref = new
    return c, abs(E)


def max_rel_err(c, grid: int = 1000001) -> float:
    xs = np.linspace(LO, HI, grid)
    return float(np.max(np.abs(np.polyval(np.asarray(c)[::-1], xs) / 2.0 ** xs - 1.0)))


if __name__ == "__main__":
    c, E = remez()
    print("coefficients c0..c3:", ", ".join(f"{v:.9g}" for v in c))
    print(f"levelled relative error {E:.4g}, max on a dense grid {max_rel_err(c):.4g}")
    c32 = np.asarray(c, dtype=np.float32).astype(np.float64)
    print(f"with fp32 coefficients: {max_rel_err(c32):.4g}")
