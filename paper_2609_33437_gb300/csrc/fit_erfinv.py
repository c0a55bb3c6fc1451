"""Fit the polynomial coefficients of the device erfinv used by the Gaussian
Perturb transform (smat_device.cuh: erfinv_poly, erfinv_poly2, erfinv_central2).

Method (structure of M. Giles, "Approximating the erfinv function", GPU
Computing Gems Jade Edition, 2011; coefficients fitted here): for
x in (-1, 1) let a = |x|, t = 1 - a^2 and L = log2(t) <= 0.
  central  (L >= L0):  erfinv(x) = x * P(L)        P a polynomial in L
  tail     (L <  L0):  erfinv(x) = x * Q(s - S_MID),  s = sqrt(-L)
The device evaluates t with one fused multiply-add, L with the hardware
log2 approximation and P, Q by Horner's rule in fp32. P is fitted on
L in [L0, 0] (P(0) = sqrt(pi) / 2), Q on s in [sqrt(-L0), sqrt(23)] (the
smallest t of an input sym(u) is 2^-23). Both fits minimise the relative
error at Chebyshev nodes with high-precision targets (mpmath).

Run: python fit_erfinv.py   (prints the coefficient tables and the error
of an fp32 Horner evaluation over every input sym() can produce).
"""

import mpmath as mp
import numpy as np

mp.mp.dps = 40
L0 = -8.0          # central / tail boundary in log2(1 - x^2)
DEG_P = 9
DEG_Q = 9
S_MAX = float(mp.sqrt(23.0)) + 1e-3
S_MID = 3.8125     # tail Horner variable s - S_MID (exact in fp32), |s - S_MID| <= 1


def f_central(L):
    """erfinv(x) / x as a function of L = log2(1 - x^2)."""
    L = mp.mpf(L)
    if L == 0:
        return mp.sqrt(mp.pi) / 2
    x = mp.sqrt(1 - mp.power(2, L))
    return mp.erfinv(x) / x


def f_tail(s):
    L = -mp.mpf(s) ** 2
    x = mp.sqrt(1 - mp.power(2, L))
    return mp.erfinv(x) / x


def fit(func, lo, hi, deg, shift=0.0, n=400):
    k = np.arange(n)
    nodes = 0.5 * (lo + hi) + 0.5 * (hi - lo) * np.cos(np.pi * (k + 0.5) / n)
    y = np.array([float(func(v)) for v in nodes])
    # relative-error least squares in the monomial basis of (variable - shift)
    V = np.vander(nodes - shift, deg + 1, increasing=True) / y[:, None]
    c, *_ = np.linalg.lstsq(V, np.ones_like(y), rcond=None)
    # a few Lawson-style reweightings toward minimax
    w = np.ones_like(y)
    for _ in range(30):
        r = V @ c - 1.0
        w = w * (np.abs(r) + 1e-30) ** 0.5
        w /= w.max()
        c, *_ = np.linalg.lstsq(V * w[:, None], w, rcond=None)
    return c  # increasing powers


def horner_f32(c, v):
    """fp32 Horner with fused multiply-adds (each step one rounding)."""
    v = np.asarray(v, np.float32)
    cc = np.asarray(c, np.float32)
    acc = np.full_like(v, cc[-1])
    for coef in cc[-2::-1]:
        acc = (acc.astype(np.float64) * v.astype(np.float64) + np.float64(coef)).astype(np.float32)
    return acc


def main():
    cP = fit(f_central, L0, 0.0, DEG_P)
    cQ = fit(f_tail, float(mp.sqrt(-L0)), S_MAX, DEG_Q, shift=S_MID)
    print("// P(L), L in [%g, 0], increasing powers" % L0)
    print("{" + ", ".join("%.9ef" % v for v in np.float32(cP)) + "}")
    print("// Q(s - %g), s = sqrt(-L) in [%g, %g], increasing powers" % (S_MID, float(mp.sqrt(-L0)), S_MAX))
    print("{" + ", ".join("%.9ef" % v for v in np.float32(cQ)) + "}")

    # error over every input sym(u) = (2k + 1 - 2^24) 2^-24, k = 2^23 .. 2^24 - 1 (x > 0)
    from scipy.special import erfinv as sp_erfinv
    k = np.arange(1 << 23, 1 << 24, dtype=np.int64)
    x = ((2 * k + 1 - (1 << 24)) * 2.0**-24).astype(np.float32)
    a = x.astype(np.float64)
    t = (1.0 - a * a).astype(np.float32)          # fma(-a, a, 1), one rounding
    L = np.log2(t.astype(np.float64)).astype(np.float32)
    ref = sp_erfinv(a)
    central = L >= np.float32(L0)
    y = np.empty_like(x)
    y[central] = (x[central].astype(np.float64) * horner_f32(cP, L[central]).astype(np.float64)).astype(np.float32)
    s = np.sqrt(-L[~central].astype(np.float64)).astype(np.float32)
    v = (s - np.float32(S_MID)).astype(np.float32)
    y[~central] = (x[~central].astype(np.float64) * horner_f32(cQ, v).astype(np.float64)).astype(np.float32)
    rel = np.abs(y.astype(np.float64) - ref) / ref
    print("max rel error: central %.3g, tail %.3g (fp32 ulp 5.96e-8); tail fraction %.4g"
          % (rel[central].max(), rel[~central].max(), (~central).mean()))
    # sensitivity to the hardware log2 (absolute error up to ~2^-22)
    for dL in (2.0**-22, -2.0**-22):
        Lp = (L.astype(np.float64) + dL).astype(np.float32)
        yc = (x[central].astype(np.float64) * horner_f32(cP, np.minimum(Lp[central], 0)).astype(np.float64))
        print("  with log2 error %+.2g: central max rel %.3g" % (dL, (np.abs(yc - ref[central]) / ref[central]).max()))


if __name__ == "__main__":
    main()
