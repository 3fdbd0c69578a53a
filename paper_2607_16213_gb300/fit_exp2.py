"""Derives the coefficients of ex2_poly (csrc/ptx.cuh): the degree-5 polynomial p(f) ~ 2^f on
[-1/2, 1/2] that minimises the maximum relative error (Remez exchange, started from a
Chebyshev-node least-squares fit), rounded to fp32, and the error of its fp32 Horner form.

    python -m paper_2607_16213_gb300.fit_exp2
"""
import numpy as np


def remez_exp2(deg: int, iters: int = 30) -> np.ndarray:
    grid = np.linspace(-0.5, 0.5, 200001)
    xs = 0.5 * np.cos(np.pi * np.arange(deg + 2) / (deg + 1))[::-1]  # initial reference
    c = None
    for _ in range(iters):
        M = np.zeros((deg + 2, deg + 2))
        for i, xi in enumerate(xs):
            M[i, :deg + 1] = xi ** np.arange(deg + 1)
            M[i, deg + 1] = (-1) ** i * np.exp2(xi)  # equioscillating relative error
        c = np.linalg.solve(M, np.exp2(xs))[:deg + 1]
        err = (np.polyval(c[::-1], grid) - np.exp2(grid)) / np.exp2(grid)
        segs = np.split(np.arange(len(grid)), np.where(np.diff(np.sign(err)) != 0)[0] + 1)
        ext = [seg[np.argmax(np.abs(err[seg]))] for seg in segs]
        if len(ext) != deg + 2:
            break
        xs = grid[ext]
    return c


def horner_f32(c32: np.ndarray, f: np.ndarray) -> np.ndarray:
    p = np.full_like(f, c32[-1])
    for k in range(len(c32) - 2, -1, -1):
        p = (p * f + c32[k]).astype(np.float32)
    return p


if __name__ == "__main__":
    c32 = remez_exp2(5).astype(np.float32)
    f = np.linspace(-0.5, 0.5, 100001).astype(np.float32)
    rel = np.abs(horner_f32(c32, f).astype(np.float64) / np.exp2(f.astype(np.float64)) - 1.0).max()
    print("coefficients (c0..c5):", ", ".join("%.8e" % v for v in c32))
    print("max relative error of the fp32 Horner form: %.3g" % rel)
