"""Host-side pins of closed-form approximations the kernels use (no GPU needed).

The GEMM epilogue and the surrogate heads compute GELU's erf with Abramowitz & Stegun,
Handbook of Mathematical Functions (1964), formula 7.1.26, whose stated absolute error
bound is 1.5e-7.  Restating the formula with the constants the kernels use and checking
that bound against scipy's erf catches a mistyped constant."""
import numpy as np
import scipy.special

P = 0.3275911
A = (0.254829592, -0.284496736, 1.421413741, -1.453152027, 1.061405429)


def erf_as(x):
    ax = np.abs(x)
    t = 1.0 / (1.0 + P * ax)
    poly = t * (A[0] + t * (A[1] + t * (A[2] + t * (A[3] + t * A[4]))))
    return np.sign(x) * (1.0 - poly * np.exp(-ax * ax))


def test_erf_7_1_26_within_its_bound():
    x = np.linspace(-8, 8, 200001)
    assert np.max(np.abs(erf_as(x) - scipy.special.erf(x))) <= 1.5e-7


def test_gelu_from_7_1_26_matches_exact_gelu():
    x = np.linspace(-10, 10, 100001)
    g = 0.5 * x * (1.0 + erf_as(x / np.sqrt(2.0)))
    exact = 0.5 * x * (1.0 + scipy.special.erf(x / np.sqrt(2.0)))
    assert np.max(np.abs(g - exact)) <= 1.5e-7 * 0.5 * 10


def test_packed_gelu_form_matches_exact_gelu():
    """The packed-pair GELU of the GEMM epilogue and the surrogate heads rewrites
    x (1 + erf(x / sqrt 2)) as x + |x| r with r = 1 - poly(t) e^{-x^2 / 2} (7.1.26, t = 1 /
    (1 + p |x| / sqrt 2)), evaluates poly with negated coefficients and forms e^{-x^2/2} as
    2^(-log2(e) / 2 x^2); simulated here step by step in float32."""
    f = np.float32
    x = np.linspace(-10, 10, 200001).astype(f)
    ax = np.abs(x)
    d = (ax * f(P * 0.70710678118654752) + f(1)).astype(f)
    t = (f(1) / d).astype(f)
    p = (t * f(-A[4]) + f(-A[3])).astype(f)
    p = (t * p + f(-A[2])).astype(f)
    p = (t * p + f(-A[1])).astype(f)
    p = (t * p + f(-A[0])).astype(f)
    p = (p * t).astype(f)
    q = (ax * (ax * f(-0.5 * 1.4426950408889634))).astype(f)
    e = np.exp2(q.astype(np.float64)).astype(f)
    r = (p * e + f(1)).astype(f)
    g = ((ax * r + x) * f(0.5)).astype(np.float64)
    xd = x.astype(np.float64)
    exact = 0.5 * xd * (1.0 + scipy.special.erf(xd / np.sqrt(2.0)))
    # float32 evaluation adds a few ulps of |x| to the formula's own 1.5e-7 bound
    assert np.all(np.abs(g - exact) <= 1.5e-7 * 0.5 * np.abs(xd) + 4e-7 * np.abs(xd) + 1e-12)
