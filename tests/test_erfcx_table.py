"""The device erfcx's polynomial (sdv_device.cuh) is the one the committed generator
prints, and the generator's fit meets its stated accuracy (CPU only)."""
import os
import re
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2606_13426_gb300", "csrc")
sys.path.insert(0, CSRC)
import gen_erfcx_coeffs as G  # noqa: E402


def _device_coefficients():
    src = open(os.path.join(CSRC, "sdv_device.cuh")).read()
    body = src[src.index("float erfcx_pos(float z)"):src.index("// erfcx of any sign")]
    lead = float(re.search(r"float f = ([-0-9.e+]+)f;", body).group(1))
    rest = [float(v) for v in re.findall(r"f = fmaf\(f, x, ([-0-9.e+]+)f\);", body)]
    return np.array([lead] + rest)[::-1]       # power basis, constant term first


def test_device_table_is_the_generators():
    dev = _device_coefficients()
    gen = G.coefficients()
    assert len(dev) == G.DEG + 1
    np.testing.assert_allclose(dev, gen, rtol=2e-8, atol=1e-12)


def test_fit_accuracy():
    assert G.max_relative_error(_device_coefficients()) < 2e-7
