"""The polynomial exponential of the block-mask kernel (block_attn.cu): its
coefficients are the ones exp2_poly.py fits, and the kernel's evaluation --
round-to-nearest split through x + 1.5 * 2^23, degree-3 Horner in fp32, the
integer part added to the exponent field -- stays within 1e-4 relative of 2^x
over the range the kernel feeds it (re-evaluated here in numpy float32)."""
import importlib.util
import os
import re

import numpy as np

CSRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "paper_2402_02082_gb300", "csrc")


def _fit_module():
    spec = importlib.util.spec_from_file_location("exp2_poly", os.path.join(CSRC, "exp2_poly.py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _kernel_coefficients():
    src = open(os.path.join(CSRC, "block_attn.cu")).read()
    vals = {k: float(v) for k, v in re.findall(r"kExpC(\d) = ([0-9.eE+-]+)f", src)}
    return np.array([vals[str(i)] for i in range(4)])


def kernel_exp2(x):
    """The kernel's exp2_poly2, element by element, in float32."""
    x = np.maximum(np.asarray(x, np.float32), np.float32(-126.0))
    c = _kernel_coefficients().astype(np.float32)
    rnd = np.float32(12582912.0)
    j = (x + rnd).astype(np.float32)
    n = (j - rnd).astype(np.float32)
    f = (x - n).astype(np.float32)
    q = (c[3] * f + c[2]).astype(np.float32)
    q = (q * f + c[1]).astype(np.float32)
    q = (q * f + c[0]).astype(np.float32)
    bits = q.view(np.uint32) + (j.view(np.uint32) << np.uint32(23))
    return bits.astype(np.uint32).view(np.float32)


def test_coefficients_are_the_fit():
    c, err = _fit_module().fit()
    assert err < 1e-4
    assert np.allclose(_kernel_coefficients(), c, rtol=0, atol=5e-9)


def test_evaluation_matches_exp2():
    x = np.concatenate([np.linspace(-125.0, 8.0, 400001), np.arange(-125, 9) + 0.5, np.arange(-125, 9).astype(float)])
    got = kernel_exp2(x).astype(np.float64)
    want = np.exp2(x.astype(np.float32).astype(np.float64))
    assert np.max(np.abs(got - want) / want) < 1e-4


def test_masked_and_tiny_arguments_stay_tiny_and_positive():
    got = kernel_exp2(np.array([-np.inf, -1e30, -200.0, -126.0], np.float32))
    assert np.all(got > 0) and np.all(got < 1.2e-38 * 1.001)
