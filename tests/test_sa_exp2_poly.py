"""The polynomial exp2 of the softmax-attention kernel (csrc/gbla_sa.cu,
exp2_poly2), emulated step by step in fp32 on the CPU from the constants in
the source: its relative error against 2^x stays within the bound its comment
states, over the whole range the kernel feeds it (x <= 2^3 with the lazy
maximum; clamped at -125)."""
import os
import re

import numpy as np

SRC = os.path.join(os.path.dirname(__file__), "..", "paper_2606_07317_gb300", "csrc", "gbla_sa.cu")


def _coefficients():
    text = open(SRC).read()
    body = text[text.index("float2 exp2_poly2("):]
    body = body[:body.index("\n}\n")]
    vals = [float(v) for v in re.findall(r"make_float2\(([0-9.]+)f, \1f\)", body)]
    # Horner order in the source: c3, c2, then c1, then c0
    assert len(vals) == 4, vals
    return [np.float32(v) for v in vals]


def _fma32(a, b, c):
    return (a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64)).astype(np.float32)


def _exp2_poly(x):
    c3, c2, c1, c0 = _coefficients()
    x = np.maximum(x.astype(np.float32), np.float32(-125.0))
    k = np.float32(12582912.0)
    t = (x + k).astype(np.float32)
    r = (t - k).astype(np.float32)
    f = _fma32(r, np.full_like(r, -1.0), x)
    q = _fma32(np.full_like(f, c3), f, np.full_like(f, c2))
    q = _fma32(q, f, np.full_like(f, c1))
    q = _fma32(q, f, np.full_like(f, c0))
    bits = q.view(np.int32) + (t.view(np.int32) << 23)
    return bits.view(np.float32)


def test_exp2_poly_relative_error_bound():
    x = np.concatenate([np.linspace(-125.0, 8.0, 400001, dtype=np.float32),
                        np.linspace(-1.0, 1.0, 100001, dtype=np.float32)])
    got = _exp2_poly(x).astype(np.float64)
    ref = np.exp2(x.astype(np.float64))
    rel = np.abs(got - ref) / ref
    assert rel.max() <= 8e-5, rel.max()
    # far below the 2^-9 relative rounding every probability gets as bf16
    assert rel.max() < 2.0 ** -13


def test_exp2_poly_clamps_minus_infinity():
    # keys past the end score -inf: the value is 2^-125 (times p(0)), not NaN
    got = _exp2_poly(np.array([-np.inf, -1e30, -200.0], dtype=np.float32))
    want = _exp2_poly(np.array([-125.0], dtype=np.float32))[0]
    assert np.all(got == want) and 0 < want < 2.0 ** -124
