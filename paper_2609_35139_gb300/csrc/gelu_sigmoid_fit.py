"""Coefficients of the branch-free GELU used by the GEMM epilogue (cr_gemm.cu).

GELU(x) = x Phi(x), with Phi the standard normal CDF.  Write Phi as a logistic
function of its log2-odds, Phi(x) = 1 / (1 + 2^(-G(x))) with
G(x) = log2(Phi(x) / (1 - Phi(x))), an odd function of x.  The epilogue uses

    Phi(x) ~ 1 / (1 + 2^(x H(x^2)))        (H fitted to -G(x) / x)

with H a polynomial of degree DEG in s = x^2, so that one GELU costs a square,
DEG fused multiply-adds, a multiply, one 2^y, an add, one reciprocal and the
final multiply.  H is fitted on x in (0, X] by least squares on Chebyshev nodes,
weighted by the sensitivity of GELU to G (x Phi (1 - Phi) ln 2), then refined by
Lawson's iteration towards the minimax absolute error of GELU.  Beyond X the
same formula holds without a clamp: H(s) <= H(0) < 0 for every s >= 0 and
|x H(x^2)| >= 34 for |x| >= X (check() verifies both), so the approximate Phi
is within 2^-34 of 0 or 1 there, as the exact one is within 1e-9.

Run: python gelu_sigmoid_fit.py  -> prints the coefficients h0 .. h6 and the
error figures of check() in float64.
"""
import numpy as np
from scipy.special import erfc, log_ndtr, ndtr

DEG = 6
X = 6.0
LOG2E = 1.0 / np.log(2.0)


def log2_odds(x):
    """G(x) = log2(Phi(x) / (1 - Phi(x))), stable in both tails."""
    return (log_ndtr(x) - log_ndtr(-x)) * LOG2E


def fit():
    n = 20000
    k = np.arange(n)
    x = X * 0.5 * (1.0 + np.cos(np.pi * (k + 0.5) / n))     # Chebyshev nodes of (0, X)
    s = x * x
    h = -log2_odds(x) / x
    w = x * ndtr(x) * ndtr(-x) * np.log(2.0) + 1e-4 * ndtr(x) * ndtr(-x)
    V = np.vander(s, DEG + 1, increasing=True)
    lw = np.ones_like(x)
    for _ in range(30):                         # Lawson: reweight by the error
        ww = w * np.sqrt(lw)
        c, *_ = np.linalg.lstsq(V * ww[:, None], h * ww, rcond=None)
        e = np.abs(w * (V @ c - h))
        lw = lw * e / e.sum()
        lw = np.maximum(lw, 1e-30)
    return c


def gelu(x, c):
    """The epilogue's formula in float64."""
    with np.errstate(over="ignore"):
        return x / (1.0 + np.exp2(x * np.polynomial.polynomial.polyval(x * x, c)))


def gelu_exact(x):
    # x/2 (1 + erf(x / sqrt 2)) as x/2 erfc(-x / sqrt 2): no cancellation in the tail
    return 0.5 * x * erfc(-x / np.sqrt(2.0))


def check(c):
    """(max |error| on [-12, 12], max error relative to |GELU| for |x| <= 3,
    the smallest |x H(x^2)| for |x| >= X, the largest H on s >= 0)."""
    x = np.linspace(-12.0, 12.0, 960001)
    ref = gelu_exact(x)
    err = np.abs(gelu(x, c) - ref)
    m = (np.abs(x) <= 3.0) & (x != 0.0)
    rel = float(np.max(err[m] / np.abs(ref[m])))
    xt = np.concatenate([np.linspace(X, 100.0, 100000), np.geomspace(100.0, 1e18, 1000)])
    tail = float(np.min(np.abs(xt * np.polynomial.polynomial.polyval(xt * xt, c))))
    s = np.concatenate([np.linspace(0.0, 1e4, 100001), np.geomspace(1e4, 1e36, 1000)])
    hmax = float(np.max(np.polynomial.polynomial.polyval(s, c)))
    return float(err.max()), rel, tail, hmax


if __name__ == "__main__":
    c = fit()
    for i, v in enumerate(c):
        print(f"h{i} = {v:.9e}")
    print("max abs error, max rel error |x|<=3, min |x H| for |x|>=X, max H:", check(c))
