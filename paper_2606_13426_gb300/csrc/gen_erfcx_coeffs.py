"""Coefficients of the device erfcx (sdv_device.cuh: erfcx_pos).

The scaled complementary error function erfcx(z) = exp(z^2) erfc(z) of z >= 0 is
written, in the variable t = 1/(1 + z/2) in (0, 1] (the substitution of Press et al.'s
erfc approximation, Numerical Recipes sec. 6.2), as erfcx(z) = t exp(f(t)), where
f(t) = log(erfcx(z)/t) is smooth on [0, 1] (f(1) = 0; f(0) = -log(2 sqrt(pi))).  f is
fitted here by a Chebyshev least-squares fit of degree 11 on Chebyshev nodes of
x = 2t - 1 (scipy's erfcx in fp64 as the reference), converted to the power basis in
x for Horner evaluation in fp32.  Run it to print the table:

    python gen_erfcx_coeffs.py
"""
import numpy as np
from numpy.polynomial import chebyshev as C
from scipy.special import erfcx

DEG = 11


def coefficients(deg=DEG, n=6000):
    x = np.cos(np.pi * (np.arange(n) + 0.5) / n)          # Chebyshev nodes of [-1, 1]
    t = 0.5 * (x + 1.0)
    keep = t > 1e-12
    x, t = x[keep], t[keep]
    z = 2.0 * (1.0 - t) / t
    f = np.log(erfcx(z) / t)
    return C.cheb2poly(C.chebfit(x, f, deg))              # power basis in x


def max_relative_error(p, n=400001):
    """fp32 Horner evaluation of t exp(f) against scipy's erfcx, over t in (0, 1]."""
    t = np.linspace(1e-6, 1.0, n)
    x = (2.0 * t - 1.0).astype(np.float32)
    acc = np.float32(p[-1])
    for c in p[-2::-1]:
        acc = (acc * x + np.float32(c)).astype(np.float32)
    z = 2.0 * (1.0 - t) / t
    return float(np.max(np.abs(t * np.exp(acc.astype(np.float64)) / erfcx(z) - 1.0)))


if __name__ == "__main__":
    p = coefficients()
    print("// f(t) = log(erfcx(z)/t), t = 1/(1 + z/2), power basis in x = 2t - 1, degree %d" % DEG)
    print("// (max relative error of t exp(f) with fp32 Horner: %.2e)" % max_relative_error(p))
    print("constexpr float kErfcxP[%d] = {" % (DEG + 1))
    print(",\n".join("    %.9ef" % c for c in p) + "};")
