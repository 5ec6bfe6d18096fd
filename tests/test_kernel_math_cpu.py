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
