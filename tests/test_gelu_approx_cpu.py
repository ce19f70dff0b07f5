"""The erf approximation the bf16 tensor-core epilogues use for the exact GELU
(Hastings, Abramowitz & Stegun formula 7.1.26), checked against math.erf over the
whole range against its published bound |error| <= 1.5e-7, together with the
GELU and GELU' built from it against their closed forms.  (The GPU parity tests
check the kernels' H, A and dH outputs against the fp64 oracle.)"""
import math

import numpy as np

P, A1, A2, A3, A4, A5 = 0.3275911, 0.254829592, -0.284496736, 1.421413741, -1.453152027, 1.061405429


def phi_parts(h):
    x = np.abs(h) / math.sqrt(2.0)
    t = 1.0 / (1.0 + P * x)
    poly = t * (A1 + t * (A2 + t * (A3 + t * (A4 + t * A5))))
    E = np.exp(-0.5 * h * h)
    tail = 0.5 * poly * E
    return np.where(h >= 0, 1.0 - tail, tail), E


def test_hastings_erf_bound():
    x = np.linspace(0.0, 8.0, 200001)
    t = 1.0 / (1.0 + P * x)
    approx = 1.0 - t * (A1 + t * (A2 + t * (A3 + t * (A4 + t * A5)))) * np.exp(-x * x)
    exact = np.array([math.erf(v) for v in x])
    assert np.max(np.abs(approx - exact)) <= 1.5e-7


def test_gelu_and_derivative_from_the_approximation():
    h = np.linspace(-12.0, 12.0, 100001)
    Phi, E = phi_parts(h)
    exact_Phi = 0.5 * (1.0 + np.array([math.erf(v / math.sqrt(2.0)) for v in h]))
    exact_phi = np.exp(-0.5 * h * h) / math.sqrt(2.0 * math.pi)
    gelu = h * Phi
    dgelu = Phi + h * E / math.sqrt(2.0 * math.pi)
    assert np.max(np.abs(gelu - h * exact_Phi) / np.maximum(1.0, np.abs(h))) <= 1.0e-7
    assert np.max(np.abs(dgelu - (exact_Phi + h * exact_phi))) <= 1.0e-7
