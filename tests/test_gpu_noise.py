"""GPU unit noise transforms against their definitions: sym(w) bit-exact over
all 2^24 inputs; the device erfinv (fitted polynomials, fit_erfinv.py)
within 5e-7 relative of the oracle's erfinv (Newton in double) on every 8th
input and on every input of the tail region, exactly odd, and monotone; the
Laplace transform -sign(v) ln(1 - |v|) within 3 fp32 ulps of the oracle's
double on all 2^24 inputs, exactly odd, and monotone."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S

pytestmark = pytest.mark.gpu

ERFINV_RTOL = 5e-7


def _words(k):
    return torch.from_numpy((np.asarray(k, np.int64) << 8).astype(np.uint32).view(np.int32)).cuda()


def test_uniform_unit_transform_exact_all_inputs():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    k = np.arange(1 << 24, dtype=np.int64)
    got = S.debug_noise_unit(_words(k), S.SMAT_NOISE_UNIFORM).cpu().numpy()
    ref = ((2 * k + 1 - (1 << 24)) * 2.0**-24).astype(np.float32)
    assert np.array_equal(got.view(np.uint32), ref.view(np.uint32))


def test_gaussian_unit_transform_accuracy_oddness_monotonicity():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    k_all = np.arange(1 << 24, dtype=np.int64)
    z = S.debug_noise_unit(_words(k_all), S.SMAT_NOISE_GAUSSIAN).cpu().numpy().astype(np.float64)
    x = (2 * k_all + 1 - (1 << 24)) * 2.0**-24
    # exactly odd: input k and 2^24 - 1 - k are negatives of each other
    assert np.array_equal(z, -z[::-1])
    # monotone non-decreasing in the input
    assert np.all(np.diff(z) >= 0)
    # accuracy against the oracle's erfinv
    pos = k_all >= (1 << 23)
    sel = pos & ((k_all % 8 == 0) | (np.abs(x) > 0.996))
    ref = O.erfinv(x[sel])
    rel = np.abs(z[sel] - ref) / np.abs(ref)
    assert rel.max() <= ERFINV_RTOL, float(rel.max())


def test_laplace_unit_transform_accuracy_oddness_monotonicity():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    k_all = np.arange(1 << 24, dtype=np.int64)
    z = S.debug_noise_unit(_words(k_all), S.SMAT_NOISE_LAPLACE).cpu().numpy()
    x = (2 * k_all + 1 - (1 << 24)) * 2.0**-24
    z64 = z.astype(np.float64)
    assert np.array_equal(z64, -z64[::-1])
    assert np.all(np.diff(z64) >= 0)
    ref = O.laplace(x)
    # within 3 ulps of the double value (log1pf and one rounding of the result)
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(z64 - ref) / ulp) <= 3.0
