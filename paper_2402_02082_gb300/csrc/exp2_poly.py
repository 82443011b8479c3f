"""Writes the coefficients of the degree-3 polynomial that the block-mask
attention kernel (block_attn.cu) uses for part of its exponentials.

2^f on [-1/2, 1/2] by a relative-error minimax fit (Remez exchange on the
linear system p(x_i) - 2^x_i = (-1)^i E 2^x_i over d + 2 alternation points,
starting from Chebyshev extrema).  Run: python exp2_poly.py
"""
import numpy as np


def fit(degree=3, iters=30, grid=200001):
    """Coefficients c_0..c_d (ascending) and the max relative error on the grid."""
    a, b = -0.5, 0.5
    k = np.arange(degree + 2)
    x = 0.5 * (a + b) + 0.5 * (b - a) * np.cos(np.pi * (degree + 1 - k) / (degree + 1))
    g = np.linspace(a, b, grid)
    c = None
    for _ in range(iters):
        A = np.zeros((degree + 2, degree + 2))
        for i, xi in enumerate(x):
            A[i, :degree + 1] = xi ** np.arange(degree + 1)
            A[i, degree + 1] = (-1) ** i * 2.0 ** xi
        c = np.linalg.solve(A, 2.0 ** x)[:degree + 1]
        err = (np.polyval(c[::-1], g) - 2.0 ** g) / 2.0 ** g
        turn = [0] + [i for i in range(1, grid - 1) if (err[i] - err[i - 1]) * (err[i + 1] - err[i]) <= 0] + [grid - 1]
        if len(turn) != degree + 2:
            break
        x = g[turn]
    err = (np.polyval(c[::-1], g) - 2.0 ** g) / 2.0 ** g
    return c, float(np.abs(err).max())


if __name__ == "__main__":
    c, e = fit()
    print("coefficients (ascending):", ", ".join(f"{float(v):.9g}f" for v in c))
    print("max relative error:", e)
