"""Coefficients of the degree-3 polynomial that exp2_poly2 (ptx_sm103.cuh) uses
for 2^f on [-1/2, 1/2]: the minimax fit of relative error, by the Remez
exchange algorithm. Prints the coefficients (c0..c3, rounded to fp32) and the
maximum relative error of the fp32 Horner evaluation."""

import numpy as np


def remez(deg, a=-0.5, b=0.5, iters=30, grid=200001):
    n = deg + 2
    x = 0.5 * (a + b) + 0.5 * (b - a) * np.cos(np.pi * np.arange(n)[::-1] / (n - 1))
    g = np.linspace(a, b, grid)
    for _ in range(iters):
        y = 2.0 ** x
        A = np.zeros((n, n))
        A[:, : deg + 1] = x[:, None] ** np.arange(deg + 1)
        A[:, deg + 1] = (-1.0) ** np.arange(n) * y
        c = np.linalg.solve(A, y)[: deg + 1]
        err = (np.polyval(c[::-1], g) - 2.0 ** g) / 2.0 ** g
        runs = np.split(np.arange(grid), np.where(np.diff(np.sign(err)) != 0)[0] + 1)
        ext = [r[np.argmax(np.abs(err[r]))] for r in runs]
        if len(ext) == n:
            x = g[ext]
    return c


def main(deg=3):
    c = remez(deg).astype(np.float32)
    f = np.linspace(-0.5, 0.5, 1000001).astype(np.float32)
    p = np.float32(c[deg])
    for k in range(deg - 1, -1, -1):
        p = (p * f + c[k]).astype(np.float32)
    ref = 2.0 ** f.astype(np.float64)
    print("coefficients", [float(v) for v in c])
    print("max relative error", float(np.abs((p - ref) / ref).max()))


if __name__ == "__main__":
    main()
