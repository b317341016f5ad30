"""Derives the coefficients of the FMA-pipe 2^f polynomial used by the
tensor-core attention kernel (prefill.cu, poly_exp2).

2^f on [-0.5, 0.5] by a cubic that minimises the maximum relative error:
Lawson's algorithm (iteratively reweighted least squares converging to the
minimax fit) on 2001 Chebyshev nodes.  Prints the fp32 coefficients and the
maximum relative error of the fp32 Horner evaluation (about 7.5e-5, far below
the 2^-9 rounding step of the bf16 probabilities it produces).
"""
import numpy as np


def fit(degree=3, nodes=2001, rounds=200):
    k = np.arange(nodes)
    f = 0.5 * np.cos(np.pi * (k + 0.5) / nodes)
    y = 2.0 ** f
    A = np.vstack([f ** i for i in range(degree + 1)]).T
    w = np.ones(nodes)
    for _ in range(rounds):
        W = np.sqrt(w) / y
        c, *_ = np.linalg.lstsq(A * W[:, None], y * W, rcond=None)
        err = np.abs(A @ c / y - 1)
        w = w * err
        w /= w.sum()
    return c.astype(np.float32)


def max_rel_error(c):
    f = np.linspace(-0.5, 0.5, 200001).astype(np.float32)
    p = np.zeros_like(f)
    for ci in c[::-1]:
        p = (p * f + ci).astype(np.float32)
    return float(np.max(np.abs(p.astype(np.float64) / 2.0 ** f.astype(np.float64) - 1)))


if __name__ == "__main__":
    c = fit()
    print("coefficients c0..c3:", [float(x) for x in c])
    print("max relative error:", max_rel_error(c))
