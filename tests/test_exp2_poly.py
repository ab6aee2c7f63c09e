"""The cubic the attention kernel may use for part of its exponentials
(2^x = 2^round(x) * p(x - round(x))): its coefficients are re-derived here by
a weighted least-squares fit of the relative error on [-1/2, 1/2] (Lawson
iterations on Chebyshev nodes), and the composed 2^x is checked in float32
arithmetic against the exact value (no GPU)."""
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def fit_cubic():
    n = 2001
    f = 0.5 * np.cos(np.pi * (np.arange(n) + 0.5) / n)
    y = 2.0 ** f
    a = np.vander(f, 4, increasing=True)
    w = np.ones(n)
    for it in range(200):
        wt = w / y
        c, *_ = np.linalg.lstsq(a * wt[:, None], y * wt, rcond=None)
        e = np.abs(a @ c - y) / y
        if it < 199:
            w = w * (e / e.max()) ** 0.2
            w /= w.sum()
    return c


def kernel_coefficients():
    src = open(os.path.join(ROOT, "paper_2607_27600_gb300", "csrc", "attn.cu")).read()
    body = src[src.index("CC_DEV float2 exp2_poly2"):]
    body = body[:body.index("return make_float2")]
    vals = [float(v) for v in re.findall(r"make_float2\(([0-9.e+-]+)f,", body)]
    # order in the Horner evaluation: c3, c2, c1, c0
    return np.array([vals[3], vals[2], vals[1], vals[0]])


def test_coefficients_are_the_fit():
    np.testing.assert_allclose(kernel_coefficients(), fit_cubic(), rtol=1e-6, atol=1e-7)


def test_composed_exp2_float32():
    c = kernel_coefficients().astype(np.float32)
    x = np.concatenate([np.linspace(-125, 8, 400001), [-0.5, 0.5, 0.0, 7.99]]).astype(np.float32)
    magic = np.float32(12582912.0)
    t = (x + magic).astype(np.float32)
    j = (t - magic).astype(np.float32)
    f = (x - j).astype(np.float32)
    p = ((c[3] * f + c[2]) * f + c[1]) * f + c[0]
    p = p.astype(np.float32)
    bits = (p.view(np.uint32).astype(np.uint64) + (t.view(np.uint32).astype(np.uint64) << 23)) & 0xFFFFFFFF
    got = bits.astype(np.uint32).view(np.float32).astype(np.float64)
    want = 2.0 ** x.astype(np.float64)
    assert np.all(np.abs(f) <= 0.5)
    assert np.max(np.abs(got - want) / want) < 1e-4
