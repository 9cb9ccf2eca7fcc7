"""The branch-free GELU of the GEMM epilogue: its coefficients are the ones the
committed fit script produces, the formula meets its error bounds against the
definition GELU(x) = x/2 (1 + erf(x / sqrt 2)), in float64 and evaluated in
float32 the way the kernel does, and it behaves in the tails.  No GPU needed."""
import importlib.util
import math
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_35139_gb300", "csrc")


def _fit_module():
    spec = importlib.util.spec_from_file_location("gelu_sigmoid_fit",
                                                  os.path.join(CSRC, "gelu_sigmoid_fit.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _kernel_coefficients():
    with open(os.path.join(CSRC, "cr_gemm.cu")) as f:
        src = f.read()
    body = re.search(r"kGeluH\[7\]\s*=\s*\{([^}]*)\}", src).group(1)
    return np.array([float(v.strip().rstrip("f")) for v in body.split(",") if v.strip()])


def _definition(x):
    # math.erf, independent of the scipy routines the fit uses
    return np.array([0.5 * v * (1.0 + math.erf(v / math.sqrt(2.0))) for v in x])


def test_kernel_coefficients_are_the_fit():
    m = _fit_module()
    k = _kernel_coefficients()
    assert k.shape == (m.DEG + 1,) == (7,)
    np.testing.assert_allclose(k, m.fit(), rtol=1e-8, atol=1e-15)


def test_fit_error_bounds_and_tails():
    m = _fit_module()
    err, rel, tail, hmax = m.check(_kernel_coefficients())
    assert err < 1e-7            # absolute, over [-12, 12]
    assert rel < 2e-5            # relative to |GELU| for |x| <= 3
    assert tail > 30.0           # |x H(x^2)| for |x| >= 6: Phi within 2^-30 of 0 or 1
    assert hmax < -2.0           # H < 0 on s >= 0: the log2-odds keep the sign of x


def test_formula_against_definition():
    m = _fit_module()
    c = _kernel_coefficients()
    x = np.concatenate([np.linspace(-10.0, 10.0, 2001), [-1e-3, 1e-3, -0.5, 0.5, 0.0]])
    ref = _definition(x)
    np.testing.assert_allclose(m.gelu(x, c), ref, rtol=0, atol=1e-7)
    # known values: GELU(0) = 0, GELU(1) = Phi(1) = 0.841344746..., odd part x/2
    assert m.gelu(np.array([0.0]), c)[0] == 0.0
    assert abs(m.gelu(np.array([1.0]), c)[0] - 0.8413447460685429) < 1e-7
    g = m.gelu(np.array([2.5, -2.5]), c)
    assert abs((g[0] - g[1]) - 2.5) < 2e-7      # GELU(x) - GELU(-x) = x


def test_float32_evaluation():
    """The kernel's operation order in float32 (square, Horner, multiply, 2^y, add,
    reciprocal, multiply; 2^y and 1/y taken exact in float32)."""
    c = _kernel_coefficients().astype(np.float32)
    x = np.linspace(-12.0, 12.0, 200001).astype(np.float32)
    s = x * x
    h = np.full_like(x, c[6])
    for i in range(5, -1, -1):
        h = (h * s + c[i]).astype(np.float32)
    with np.errstate(over="ignore"):
        e = np.exp2(h * x).astype(np.float32)
    g = (x * (np.float32(1.0) / (e + np.float32(1.0)))).astype(np.float32)
    ref = 0.5 * x.astype(np.float64) * (1.0 + np.vectorize(math.erf)(x.astype(np.float64) / math.sqrt(2.0)))
    err = np.abs(g.astype(np.float64) - ref)
    assert np.all(np.isfinite(g))
    assert np.all(err <= 2e-7 + 4e-7 * np.abs(ref)), float(np.max(err - 4e-7 * np.abs(ref)))
