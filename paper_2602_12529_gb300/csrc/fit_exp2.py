"""Fits the polynomial p(f) ~ 2^f on f in [-1/2, 1/2] used by the attention
kernel's software exp2 (csrc/attention.cu), by the Remez exchange algorithm
on the relative error.  Prints the fp32 coefficients (c0 + c1 f + ...) and the
maximum relative error of the fp32-rounded polynomial.

Method: range reduction 2^x = 2^n * 2^f with n = round(x) (Cody-Waite style
split into integer and fraction), then a minimax polynomial for 2^f whose
coefficients come from this script.  Run: python fit_exp2.py [degree]
"""
import sys

import numpy as np


def remez(deg, lo=-0.5, hi=0.5, iters=30):
    f = lambda x: np.exp2(x)
    n = deg + 2
    # Chebyshev extrema as the starting reference
    x = 0.5 * (lo + hi) + 0.5 * (hi - lo) * np.cos(np.pi * np.arange(n)[::-1] / (n - 1))
    grid = np.linspace(lo, hi, 200001)
    for _ in range(iters):
        # solve p(x_i) + (-1)^i E f(x_i) = f(x_i) for the coefficients and E
        A = np.zeros((n, n))
        for i in range(n):
            A[i, :deg + 1] = x[i] ** np.arange(deg + 1)
            A[i, deg + 1] = (-1) ** i * f(x[i])
        sol = np.linalg.solve(A, f(x))
        c = sol[:deg + 1]
        err = (np.polyval(c[::-1], grid) - f(grid)) / f(grid)
        # new reference: extrema of the error between sign changes
        sign = np.sign(err)
        idx = np.concatenate([[0], np.nonzero(np.diff(sign))[0] + 1, [len(grid)]])
        ext = [s + np.argmax(np.abs(err[s:e])) for s, e in zip(idx[:-1], idx[1:])]
        if len(ext) != n:
            break
        x = grid[ext]
    return c


def main():
    deg = int(sys.argv[1]) if len(sys.argv) > 1 else 3
    c = remez(deg).astype(np.float32)
    g = np.linspace(-0.5, 0.5, 1000001, dtype=np.float32)
    p = np.zeros_like(g)
    for k in range(deg, -1, -1):
        p = (p * g + c[k]).astype(np.float32)
    rel = np.max(np.abs(p.astype(np.float64) / np.exp2(g.astype(np.float64)) - 1.0))
    for k, v in enumerate(c):
        print(f"c{k} = {float(v):.9e}f  ({float(v).hex()})")
    print(f"max relative error on [-1/2, 1/2]: {rel:.3e}")


if __name__ == "__main__":
    main()
