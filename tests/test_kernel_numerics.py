"""CPU checks of numerical methods the kernels use in place of library calls."""
import numpy as np
from scipy.special import erf


def test_published_erf_approximation_bound_used_by_the_scorer_kernel():
    """The scorer kernel evaluates GELU with Abramowitz & Stegun, formula
    7.1.26; its published bound |erf_approx - erf| <= 1.5e-7 holds (fp64)."""
    z = np.linspace(0, 8, 200001)
    t = 1.0 / (1.0 + 0.3275911 * z)
    poly = t * (0.254829592 + t * (-0.284496736 + t * (1.421413741 + t * (-1.453152027 + t * 1.061405429))))
    approx = 1.0 - poly * np.exp(-z * z)
    assert np.max(np.abs(approx - erf(z))) <= 1.5e-7
