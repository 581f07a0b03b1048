"""The fitted constants the CUDA kernels carry (no GPU needed): the erf of the
GELU epilogue is the fit its generator script produces, and that fit meets
the error bound the kernel's comment states (evaluated in fp32 as the kernel
does)."""
import importlib.util
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_21291_gb300", "csrc")


def _load(name):
    spec = importlib.util.spec_from_file_location(name, os.path.join(CSRC, name + ".py"))
    m = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(m)
    return m


def _floats(src):
    return [float(v) for v in re.findall(r"([-+]?\d\.\d+e[-+]\d+)f", src)]


def test_erf_fit_matches_kernel_and_bound():
    pytest.importorskip("scipy")
    from scipy.special import erf
    m = _load("erf_poly")
    c = m.fit()
    src = open(os.path.join(CSRC, "gemm_tcgen05.cu")).read()
    body = src[src.index("float2 erf_fit2("):src.index("float2 gelu2(")]
    kern = _floats(body)[::-1]             # Horner order: highest degree first
    assert len(kern) == len(c)
    assert np.allclose(kern, c, rtol=1e-6, atol=0)
    z = np.linspace(0, 8, 200001)
    assert np.max(np.abs(m.erf_fp32(z, c).astype(np.float64) - erf(z))) <= 3.3e-7
