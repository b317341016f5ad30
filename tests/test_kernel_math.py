"""Host-side checks of arithmetic the kernels use (CPU only).

poly_exp2_x2 (prefill.cu) computes 2^x on the FMA pipe for half of the
softmax exponentials of fully visible key tiles.  Its steps are re-evaluated here in fp32 numpy and
compared with the mathematical 2^x; the coefficients in the kernel source
must be the ones the committed fit script derives.
"""
import importlib.util
import os
import re

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2605_11232_gb300", "csrc")


def _kernel_coeffs():
    """c0..c3 as written in the kernel's Horner steps:
    p = ffma2(c3, f, c2); p = ffma2(p, f, c1); p = ffma2(p, f, c0)."""
    src = open(os.path.join(CSRC, "prefill.cu")).read()
    body = src[src.index("float2 poly_exp2_x2("):]
    body = body[: body.index("\n}\n")]
    pairs = re.findall(r"make_float2\(([0-9.]+)f, \1f\)", body)
    # order of appearance: c3, c2, c1, c0 (the 1.5*2^23 constants are not of this form)
    cs = [float(x) for x in pairs if float(x) < 2.0]
    c3, c2, c1, c0 = cs
    return np.array([c0, c1, c2, c3], np.float32), cs


def _fma32(a, b, c):
    """fp32 fused multiply-add (exact product and sum in fp64, one rounding)."""
    return (a.astype(np.float64) * b.astype(np.float64) + c.astype(np.float64)).astype(np.float32)


def _poly_exp2_f32(x, c):
    """The kernel's steps in fp32: clamp, magic-number rounding, cubic,
    exponent insertion by bits(t) * 2^23 + bits(p) modulo 2^32."""
    x = x.astype(np.float32)
    xc = np.maximum(x, np.float32(-125.0))
    t = (xc + np.float32(12582912.0)).astype(np.float32)
    n = (t - np.float32(12582912.0)).astype(np.float32)
    f = (xc - n).astype(np.float32)
    p = _fma32(np.full_like(f, c[3]), f, np.full_like(f, c[2]))
    p = _fma32(p, f, np.full_like(f, c[1]))
    p = _fma32(p, f, np.full_like(f, c[0]))
    bits = (t.view(np.uint32).astype(np.uint64) * 0x800000 + p.view(np.uint32)) & 0xFFFFFFFF
    return bits.astype(np.uint32).view(np.float32)


def test_kernel_coefficients_match_fit():
    spec = importlib.util.spec_from_file_location("fit", os.path.join(CSRC, "fit_exp2_poly.py"))
    fit = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(fit)
    want = fit.fit()
    got, _ = _kernel_coeffs()
    assert np.allclose(got, want, rtol=1e-6, atol=1e-9), (got, want)
    assert fit.max_rel_error(want) < 1e-4


def test_poly_exp2_relative_error():
    c, _ = _kernel_coeffs()
    x = np.concatenate([np.linspace(-125, 10, 400001), np.arange(-125, 11, 0.5)]).astype(np.float32)
    got = _poly_exp2_f32(x, c).astype(np.float64)
    want = np.exp2(x.astype(np.float64))
    rel = np.abs(got / want - 1)
    assert rel.max() < 1e-4, rel.max()


def test_poly_exp2_clamps_and_matches_the_exponent_trick():
    """Below -125 the result is clamped to 2^-125 (still a normal number);
    bits(t)*2^23 + bits(p) equals bits(p) + (round(x) << 23)."""
    c, _ = _kernel_coeffs()
    x = np.array([-1e30, -125.5, -126.0, -300.0], np.float32)
    got = _poly_exp2_f32(x, c).astype(np.float64)
    assert np.all(np.abs(got / 2.0 ** -125 - 1) < 1e-4)
    assert _poly_exp2_f32(np.array([0.0], np.float32), c)[0] == np.float32(c[0])
    xs = np.array([-100.25, -3.5, -0.4, 0.0, 2.75, 7.5], np.float32)
    t = (xs + np.float32(12582912.0)).astype(np.float32)
    n = np.round(xs).astype(np.int64)
    assert np.array_equal(((t.view(np.uint32).astype(np.int64) * 0x800000) & 0xFFFFFFFF),
                          (n << 23) & 0xFFFFFFFF)
