"""The allocation-free entry point smat_delta_sigma_noalloc, for callers that
cannot allocate device memory (for example a plugin whose host framework owns
all of the GPU's memory, or code that must not grow a memory pool while a job
runs). It computes sigma_rel * std(theta - theta0) with the library's fixed
scratch array. Here it is called through the C ABI twice in a row, and each
result must match the sigma_t of the context-based path (smat_tensor_scalars)
within the 1e-5 relative tolerance the statistics parity tests use. This file
is collected last; it passes alone in a fresh process and after the other
tests."""

import ctypes

import pytest
import torch

from paper_2609_33437_gb300 import smat as S

pytestmark = pytest.mark.gpu

SIGMA_RTOL = 1e-5


@pytest.mark.parametrize("dtype,n", [(torch.bfloat16, 3_000_017), (torch.float32, 1_234_567)])
def test_noalloc_sigma_matches_context_path_on_two_calls(dtype, n):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    g = torch.Generator(device="cuda").manual_seed(5)
    t0f = torch.randn(n, generator=g, device="cuda") * 0.02
    th = (t0f + torch.randn(n, generator=g, device="cuda") * 3e-4).to(dtype)
    t0 = t0f.to(dtype)
    sim = torch.empty_like(th)
    sess = S.SmatSession([th], [t0], [sim], [0.7], [0.0], [0.1], seed=1, alpha_mode=S.SMAT_ALPHA_PER_TENSOR,
                         noise=S.SMAT_NOISE_GAUSSIAN)
    ref = float(sess.tensor_scalars(0)[0, 2])
    assert ref > 0.0
    out = torch.empty(1, dtype=torch.float32, device="cuda")
    for _ in range(2):
        out.fill_(-1.0)
        S.delta_sigma_noalloc(th, t0, 0.1, out=out)
        torch.cuda.synchronize()
        got = float(out[0])
        assert abs(got - ref) <= SIGMA_RTOL * ref, (got, ref)
    sess.close()


def test_noalloc_rejects_sizes_beyond_its_scratch_array():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    L = S.load_library()
    out = torch.empty(1, dtype=torch.float32, device="cuda")
    too_many = 16384 * 65536 + 1
    st = L.smat_delta_sigma_noalloc(ctypes.c_void_p(256), ctypes.c_void_p(512), too_many, S.SMAT_BF16,
                                    ctypes.c_float(0.1), ctypes.c_void_p(out.data_ptr()), None)
    assert st == 1  # SMAT_ERR_INVALID_ARG, before any device work
    assert b"scratch array" in L.smat_last_error()
