"""Coefficients of the branch-free erfc used by the GELU epilogue (cr_gemm.cu).

For z >= 0 write t = 1 / (1 + z / 2), which maps [0, inf) onto (0, 1], and
erfc(z) = t * exp(f(t) - z^2).  The smooth function f(t) = ln(erfc(z) / t) + z^2
is fitted here by a degree-9 polynomial in t (least squares on Chebyshev nodes
of t, weighted to minimise the relative error of erfc).  This is the form of the
Chebyshev erfc approximation in Numerical Recipes (Press et al., Sec. 6.2), with
coefficients fitted by this script rather than copied.

Run: python gelu_erfc_fit.py   -> prints the coefficients (c0 .. c9) and the
maximum relative error of erfc over z in [0, 10] in float64.
"""
import numpy as np
from scipy.special import erfc, erfcx

DEG = 9


def fit():
    # Chebyshev nodes of t in (0, 1], mapped to z = 2 (1 - t) / t
    k = np.arange(4000)
    t = 0.5 * (1.0 + np.cos(np.pi * (k + 0.5) / k.size))
    z = 2.0 * (1.0 - t) / t
    f = np.log(erfcx(z) / t)                # erfcx(z) = exp(z^2) erfc(z): no underflow
    c = np.polynomial.polynomial.polyfit(t, f, DEG)
    return c


def max_rel_err(c):
    z = np.linspace(0.0, 10.0, 200001)   # erfc(10) = 2e-45: below that, float32 is 0
    t = 1.0 / (1.0 + 0.5 * z)
    approx = t * np.exp(np.polynomial.polynomial.polyval(t, c) - z * z)
    return float(np.max(np.abs(approx / erfc(z) - 1.0)))


if __name__ == "__main__":
    c = fit()
    for i, v in enumerate(c):
        print(f"c{i} = {v:.9e}")
    print("max relative error of erfc on [0, 10]:", max_rel_err(c))
