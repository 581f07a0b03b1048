"""Coefficients of the erf used by the GELU epilogue of gemm_tcgen05.cu.

erf(z) = 1 - exp(-z^2) R(z) for z >= 0, where R(z) = erfc(z) exp(z^2) is smooth
and slowly varying; R is approximated on [0, 4] by a degree-10 polynomial in
u = z / 4, fitted by least squares at Chebyshev nodes with weights exp(-z^2)
(so the fit minimises the error of erf itself). Beyond z = 4, erf(z) = 1 to
within 1.6e-8. The kernel evaluates R by Horner's rule in fp32; this script
prints the coefficients and the maximum error of that fp32 evaluation.

  python paper_2607_21291_gb300/csrc/erf_poly.py
"""
import numpy as np
from scipy.special import erf, erfcx

ZMAX, DEG, NODES = 4.0, 10, 6000


def fit():
    z = (np.cos(np.pi * (np.arange(NODES) + 0.5) / NODES) + 1) / 2 * ZMAX
    w = np.exp(-z * z)
    V = np.vander(z / ZMAX, DEG + 1, increasing=True)
    c, *_ = np.linalg.lstsq(V * w[:, None], erfcx(z) * w, rcond=None)
    return c.astype(np.float32)


def erf_fp32(z, c):
    z = np.minimum(np.abs(z).astype(np.float32), np.float32(ZMAX))
    u = (z * np.float32(1 / ZMAX)).astype(np.float32)
    acc = np.full_like(u, c[-1])
    for k in range(DEG - 1, -1, -1):
        acc = (acc * u + c[k]).astype(np.float32)
    return (np.float32(1) - np.exp(-(z * z)).astype(np.float32) * acc).astype(np.float32)


if __name__ == "__main__":
    c = fit()
    zz = np.linspace(0, 8, 800001)
    err = np.max(np.abs(erf_fp32(zz, c).astype(np.float64) - erf(zz)))
    print("coefficients c0..c%d (R(z) = sum c_k (z/4)^k):" % DEG)
    for k, v in enumerate(c):
        print("  c%-2d = %.9ef" % (k, v))
    print("max |erf error| of the fp32 evaluation on [0, 8]: %.2e" % err)
