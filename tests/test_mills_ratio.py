"""The rational Mills-ratio fit used for neighbour CDF values (csrc/mills_ratio.h)
against scipy's ndtr, evaluated in float32 the way the kernel does (with an
exact exponential; the kernel's fast exponential adds ~1e-6 relative)."""
import os
import re

import numpy as np
from scipy.special import ndtr

H = os.path.join(os.path.dirname(os.path.dirname(__file__)), "paper_2602_20427_gb300", "csrc", "mills_ratio.h")


def coeffs(name):
    txt = open(H).read()
    body = re.search(name + r"\[\d+\] = \{([^}]*)\}", txt).group(1)
    return [np.float32(float(c.strip().rstrip("f"))) for c in body.split(",")]


def test_mills_ratio_cdf_accuracy():
    P, Q = coeffs("kMillsP"), coeffs("kMillsQ")
    z = np.linspace(-12, 12, 240001).astype(np.float32)
    x = np.abs(z)
    num = P[4]
    for c in P[3::-1]:
        num = num * x + c
    den = Q[5]
    for c in Q[4::-1]:
        den = den * x + c
    q = (np.exp(-0.5 * z.astype(np.float64) ** 2) * (num / den).astype(np.float64))
    cdf = np.where(z <= 0, q, 1.0 - q)
    ref = ndtr(z.astype(np.float64))
    assert np.max(np.abs(cdf - ref)) < 2e-7
    tail = ndtr(-np.abs(z.astype(np.float64)))       # upper tail Q(|z|) without cancellation
    mask = tail > 1e-30
    assert np.max(np.abs(q[mask] / tail[mask] - 1)) < 1e-6
