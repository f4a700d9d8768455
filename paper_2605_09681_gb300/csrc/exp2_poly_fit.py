"""Coefficients of the polynomial exp2 used for part of the softmax exponentials.

Method: Cody-Waite style range reduction x = n + f with n = round(x), f in [-1/2, 1/2],
2^x = 2^n * p(f), where p is a degree-3 polynomial fitted to 2^f by minimising the maximum
relative error (Lawson's iteratively reweighted least squares on Chebyshev nodes).  The
attention rounds P to bf16 (relative step 2^-8), so a relative error near 1e-4 is ample.
Run: python exp2_poly_fit.py  -> prints the coefficients and the max relative error.
"""
import numpy as np


def fit(deg=3, n=4001, iters=200):
    k = np.arange(n)
    f = 0.5 * np.cos(np.pi * (k + 0.5) / n)          # Chebyshev nodes on [-1/2, 1/2]
    y = np.exp2(f)
    V = np.vander(f, deg + 1, increasing=True) / y[:, None]   # relative-error system
    w = np.ones(n) / n
    for _ in range(iters):
        sw = np.sqrt(w)
        c, *_ = np.linalg.lstsq(V * sw[:, None], sw, rcond=None)
        err = np.abs(V @ c - 1.0)
        w = w * err
        w /= w.sum()
    fine = np.linspace(-0.5, 0.5, 200001)
    rel = np.abs(np.polyval(c[::-1], fine) / np.exp2(fine) - 1.0).max()
    return c, rel


if __name__ == "__main__":
    c, rel = fit()
    print("coefficients c0..c3:", ", ".join("%.9ef" % x for x in c))
    print("max relative error on [-1/2, 1/2]: %.3e" % rel)
