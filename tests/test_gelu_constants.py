"""The GELU constants of the kernels against the published error bound (CPU).

The feed-forward units evaluate erf with Abramowitz & Stegun's formula 7.1.26,
erf z = 1 - (a1 t + ... + a5 t^5) exp(-z^2), t = 1 / (1 + p z), |error| <= 1.5e-7
for z >= 0.  This test reads the constants as the device code spells them
(p / sqrt 2, a_i / 2, -log2(e) / 2) from the header, undoes the folding, and
checks in float64 that the formula meets that bound and that the folded form
computes x Phi(x); the constants must also equal the published table exactly
(a change in a late digit stays inside the error bound).  All of it runs before
any GPU run (tests/test_gpu_gelu.py checks the device results themselves).
"""
import math
import os
import re

import numpy as np

HEADER = os.path.join(os.path.dirname(__file__), "..", "paper_2607_20293_gb300", "csrc", "evo_internal.h")


def _constants():
    src = open(HEADER).read()
    body = src[src.index("namespace gelu_k {"):src.index("}  // namespace gelu_k")]
    num = r"(-?[0-9.]+)f"
    p = re.search(r"P = " + num + r" \* " + num, body)
    a = {int(m.group(1)): float(m.group(2))
         for m in re.finditer(r"A([1-5]) = 0\.5f \* " + num, body)}
    c = float(re.search(r"C = " + num, body).group(1))
    xmax = float(re.search(r"XMAX = " + num, body).group(1))
    return float(p.group(1)), float(p.group(2)), [a[i] for i in range(1, 6)], c, xmax


def test_constants_meet_the_published_bound():
    p, inv_sqrt2, a, c, xmax = _constants()
    assert abs(inv_sqrt2 - 1 / math.sqrt(2)) < 1e-15
    assert abs(c + math.log2(math.e) / 2) < 1e-15
    z = np.linspace(0.0, 12.0, 600001)
    t = 1.0 / (1.0 + p * z)
    poly = t * (a[0] + t * (a[1] + t * (a[2] + t * (a[3] + t * a[4]))))
    approx = 1.0 - poly * np.exp(-z * z)
    exact = np.array([math.erf(v) for v in z])
    assert float(np.max(np.abs(approx - exact))) <= 1.5e-7
    # erf(0) = 0: the coefficients sum to 1 within the bound
    assert abs(sum(a) - 1.0) <= 1.5e-7
    # beyond XMAX the Gaussian factor is below the smallest fp32 normal
    assert 2.0 ** (c * xmax * xmax) < np.finfo(np.float32).tiny


# Abramowitz & Stegun, Handbook of Mathematical Functions, formula 7.1.26
PUBLISHED_P = 0.3275911
PUBLISHED_A = [0.254829592, -0.284496736, 1.421413741, -1.453152027, 1.061405429]


def test_constants_are_the_published_ones():
    p, _, a, _, _ = _constants()
    assert p == PUBLISHED_P
    assert a == PUBLISHED_A


def test_folded_form_is_x_phi_x():
    p, inv_sqrt2, a, c, xmax = _constants()
    x = np.linspace(-xmax, xmax, 200001)
    ax = np.abs(x)
    t = 1.0 / (1.0 + p * inv_sqrt2 * ax)
    half = [0.5 * v for v in a]
    q = half[0] + t * (half[1] + t * (half[2] + t * (half[3] + t * half[4])))
    w = t * q * 2.0 ** (ax * ax * c)          # (1 - erf(|x| / sqrt 2)) / 2
    gelu = np.maximum(x, 0.0) - ax * w
    exact = np.array([0.5 * v * (1.0 + math.erf(v / math.sqrt(2))) for v in x])
    assert float(np.max(np.abs(gelu - exact) / np.maximum(1.0, np.abs(x)))) <= 0.5 * 1.5e-7 + 1e-15
