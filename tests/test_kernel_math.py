"""Host-side checks of arithmetic the kernels use (CPU only).

poly_exp2 (prefill.cu) computes 2^x on the FMA pipe for a quarter of the
softmax exponentials.  Its steps are re-evaluated here in fp32 numpy and
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
    src = open(os.path.join(CSRC, "prefill.cu")).read()
    body = src[src.index("float poly_exp2("):]
    body = body[: body.index("\n}\n")]
    nums = [float(x) for x in re.findall(r"fmaf\([^;]*?([0-9]\.[0-9]+)f", body)]
    # fmaf(c3, f, c2); fmaf(p, f, c1); fmaf(p, f, c0)
    c3c2 = re.search(r"fmaf\(([0-9.]+)f, f, ([0-9.]+)f\)", body)
    c1 = re.search(r"fmaf\(p, f, ([0-9.]+)f\);\s*p = fmaf\(p, f, ([0-9.]+)f\)", body)
    return np.array([float(c1.group(2)), float(c1.group(1)), float(c3c2.group(2)),
                     float(c3c2.group(1))], np.float32), nums


def _poly_exp2_f32(x, c):
    x = x.astype(np.float32)
    xc = np.maximum(x, np.float32(-125.0))
    t = (xc + np.float32(12582912.0)).astype(np.float32)
    n = (t - np.float32(12582912.0)).astype(np.float32)
    f = (xc - n).astype(np.float32)
    p = (c[3] * f + c[2]).astype(np.float32)
    p = (p * f + c[1]).astype(np.float32)
    p = (p * f + c[0]).astype(np.float32)
    e = ((t.view(np.int32) - 0x4B400000).astype(np.uint32) << np.uint32(23))
    r = (p.view(np.uint32) + e).view(np.float32)
    return np.where(x < -125.0, np.float32(0.0), r)


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


def test_poly_exp2_masked_and_tiny():
    c, _ = _kernel_coeffs()
    x = np.array([-np.inf, -1e30, -125.5, -126.0], np.float32)
    assert np.all(_poly_exp2_f32(x, c) == 0.0)
    assert _poly_exp2_f32(np.array([0.0], np.float32), c)[0] == np.float32(c[0])
