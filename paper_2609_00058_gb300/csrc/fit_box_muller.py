"""Coefficients of the fp32 Box-Muller transform in sv_device.cuh.

Three polynomials, each the correction after the leading term of a series,
fitted by Lawson's iteratively reweighted least squares (a minimax method)
on a dense grid, with weights that make the error relative to the final
value:

  sin(pi x) = pi x + x^3 T(x^2),     0 <= x <= 1/4, T of degree 2
  cos(pi x) = 1 + x^2 P(x^2),        0 <= x <= 1/4, P of degree 3
  ln f = 2 atanh(s) = 2 s + s^3 R(s^2),  s = (f - 1) / (f + 1),
                                     sqrt(1/2) <= f < sqrt(2), R of degree 2

and the split ln 2 = LN2_HI + LN2_LO (LN2_HI with 16 significant bits, so
e * LN2_HI is exact for |e| < 256) and pi = PI_HI + PI_LO (PI_HI = fp32(pi)).
Run it to print the constants as C; tests check that the header holds them.
"""
import numpy as np


def lawson(f, w, xs, deg, iters=300):
    basis = np.stack([xs ** k for k in range(deg + 1)], 1)
    weight = np.ones_like(xs)
    for _ in range(iters):
        sw = np.sqrt(weight)
        c, *_ = np.linalg.lstsq(basis * (sw * w)[:, None], sw * w * f, rcond=None)
        err = np.abs(w * (f - basis @ c))
        weight = weight * err
        weight /= weight.sum()
    return c, err.max()


def coefficients(points=200001):
    x = np.linspace(0.0, 0.25, points)[1:]
    y = x * x
    t, et = lawson((np.sin(np.pi * x) - np.pi * x) / x ** 3, x ** 3 / np.sin(np.pi * x), y, 2)
    p, ep = lawson((np.cos(np.pi * x) - 1.0) / y, y / np.cos(np.pi * x), y, 3)
    smax = (np.sqrt(2.0) - 1.0) / (np.sqrt(2.0) + 1.0) * 1.001
    s = np.linspace(0.0, smax, points)[1:]
    r, er = lawson((2.0 * np.arctanh(s) - 2.0 * s) / s ** 3, s ** 3 / (2.0 * np.arctanh(s)), s * s, 2)
    f32 = lambda v: [float(np.float32(a)) for a in v]
    ln2_hi = np.round(np.log(2.0) * 65536.0) / 65536.0
    pi_hi = float(np.float32(np.pi))
    return {"T": f32(t), "P": f32(p), "R": f32(r),
            "LN2_HI": float(np.float32(ln2_hi)), "LN2_LO": float(np.float32(np.log(2.0) - ln2_hi)),
            "PI_HI": pi_hi, "PI_LO": float(np.float32(np.pi - pi_hi)),
            "errors": (et, ep, er)}


if __name__ == "__main__":
    k = coefficients()
    print("// relative approximation errors: sin %.2e, cos %.2e, ln %.2e" % k["errors"])
    for name in ("T", "P", "R"):
        for i, v in enumerate(k[name]):
            print("constexpr float kBm%s%d = %.9ef;" % (name, i, v))
    for name in ("LN2_HI", "LN2_LO", "PI_HI", "PI_LO"):
        print("constexpr float kBm%s = %.9ef;" % (name.replace("_", ""), k[name]))
