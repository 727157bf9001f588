"""Coefficients of the polynomial 2^r ~ p(r), r in [-1/2, 1/2], used by the
spatial kernel to evaluate part of its exponentials on the FMA pipe.

Method: Cody-Waite style range reduction (2^x = 2^j * 2^r with j = round(x),
r = x - j) and a minimax polynomial for 2^r found with the Remez exchange
algorithm, minimising the RELATIVE error (weight 1/2^r).  The fit is done in
float64; the printed coefficients are rounded to float32 and their error is
re-measured in float32 Horner evaluation.  Run this file to regenerate the
constants pasted into spatial_tc.cu.
"""
import numpy as np


def remez_relative(deg: int, lo: float = -0.5, hi: float = 0.5, iters: int = 30):
    f = lambda x: np.exp2(x)
    n = deg + 2
    # Chebyshev extrema as the initial reference
    k = np.arange(n)
    xs = (lo + hi) / 2 + (hi - lo) / 2 * np.cos(np.pi * k[::-1] / (n - 1))
    grid = np.linspace(lo, hi, 200001)
    c = None
    for _ in range(iters):
        # solve p(x_i) + (-1)^i E f(x_i) = f(x_i)   (relative error equioscillation)
        A = np.zeros((n, n))
        for i, x in enumerate(xs):
            A[i, :deg + 1] = x ** np.arange(deg + 1)
            A[i, deg + 1] = (-1) ** i * f(x)
        sol = np.linalg.solve(A, f(xs))
        c = sol[:deg + 1]
        err = (np.polyval(c[::-1], grid) - f(grid)) / f(grid)
        # new reference: the extrema of err in each sign-alternating segment
        sign = np.sign(err)
        sign[sign == 0] = 1
        idx = np.concatenate(([0], np.nonzero(np.diff(sign))[0] + 1, [len(grid)]))
        ext = [s + np.argmax(np.abs(err[s:e])) for s, e in zip(idx[:-1], idx[1:])]
        if len(ext) < n:
            break
        # keep the n largest alternating extrema
        while len(ext) > n:
            vals = np.abs(err[ext])
            drop = 0 if vals[0] < vals[-1] else len(ext) - 1
            ext.pop(drop)
        xs = grid[ext]
    return c


def f32_horner_error(c32, n: int = 1 << 20):
    r = np.linspace(-0.5, 0.5, n).astype(np.float32)
    p = np.full_like(r, c32[-1])
    for ci in c32[-2::-1]:
        p = (p * r + ci).astype(np.float32)
    return float(np.max(np.abs(p.astype(np.float64) / np.exp2(r.astype(np.float64)) - 1.0)))


if __name__ == "__main__":
    for deg in (3, 4, 5):
        c = remez_relative(deg)
        c32 = c.astype(np.float32)
        print("degree %d: max rel err (fp32 Horner) %.3g" % (deg, f32_horner_error(c32)))
        print("  coefficients c0..c%d:" % deg, ", ".join(np.format_float_scientific(x, unique=True)
                                                     + "f" for x in c32))
