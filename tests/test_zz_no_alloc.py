"""The allocation-free entry point smat_delta_sigma_noalloc, for callers that
cannot allocate device memory (for example a plugin whose host framework owns
all of the GPU's memory, or code that must not grow a memory pool while a job
runs). It computes sigma_rel * std(theta - theta0) with the library's fixed
scratch array. Here it is called through the C ABI, twice in a row, and each
result must match both the CPU oracle's two-pass sigma_t and the sigma_t of
the context-based path (smat_tensor_scalars), within the 1e-5 relative
tolerance the statistics parity tests use; sizes below one chunk, one
element, no element and pointers that take the per-element path are covered.
This file is collected last; it passes alone in a fresh process and after
the other tests."""

import ctypes

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S

pytestmark = pytest.mark.gpu

SIGMA_RTOL = 1e-5


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def _pair(n, dtype, seed, extra=0):
    g = torch.Generator(device="cuda").manual_seed(seed)
    t0f = torch.randn(n + extra, generator=g, device="cuda") * 0.02
    th = (t0f + torch.randn(n + extra, generator=g, device="cuda") * 3e-4 + 1e-4).to(dtype)
    return th, t0f.to(dtype)


def _host(x):
    x = x.detach().cpu().contiguous()
    if x.dtype == torch.bfloat16:
        return x.view(torch.int16).numpy().view(np.uint16)
    return x.numpy()


def _oracle_sigma(th, t0, sigma_rel):
    code = O.BF16 if th.dtype == torch.bfloat16 else O.F32
    t = O.tensor(0, th.numel(), dtype=code, sigma_rel=sigma_rel)
    return O.delta_stats(t, _host(th), _host(t0))["sigma"]


@pytest.mark.parametrize("dtype,n", [(torch.bfloat16, 3_000_017), (torch.float32, 1_234_567)])
def test_noalloc_sigma_matches_oracle_and_context_path_on_two_calls(dtype, n):
    th, t0 = _pair(n, dtype, 5)
    sim = torch.empty_like(th)
    sess = S.SmatSession([th], [t0], [sim], [0.7], [0.0], [0.1], seed=1, alpha_mode=S.SMAT_ALPHA_PER_TENSOR,
                         noise=S.SMAT_NOISE_GAUSSIAN)
    ctx = float(sess.tensor_scalars(0)[0, 2])
    ref = _oracle_sigma(th, t0, 0.1)
    assert ref > 0.0
    assert abs(ctx - ref) <= SIGMA_RTOL * ref, (ctx, ref)
    out = torch.empty(1, dtype=torch.float32, device="cuda")
    for _ in range(2):
        out.fill_(-1.0)
        S.delta_sigma_noalloc(th, t0, 0.1, out=out)
        torch.cuda.synchronize()
        got = float(out[0])
        assert abs(got - ref) <= SIGMA_RTOL * ref, (got, ref)
        assert abs(got - ctx) <= SIGMA_RTOL * ref, (got, ctx)
    sess.close()


@pytest.mark.parametrize("n,offset", [(1000, 0), (65_537, 0), (70_001, 1), (4099, 3), (1, 0), (1, 1)])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_noalloc_sigma_small_ragged_and_misaligned(dtype, n, offset):
    """Fewer elements than one 2^16-element chunk, a ragged last chunk, and
    pointers offset by a few elements (not 32-byte aligned: the per-element
    path), against the oracle; one element has std 0."""
    th_b, t0_b = _pair(n, dtype, 7 + n, extra=offset)
    th, t0 = th_b[offset:], t0_b[offset:]
    ref = _oracle_sigma(th, t0, 0.25)
    out = torch.full((1,), -1.0, dtype=torch.float32, device="cuda")
    S.delta_sigma_noalloc(th, t0, 0.25, out=out)
    torch.cuda.synchronize()
    got = float(out[0])
    if n == 1:
        assert ref == 0.0 and got == 0.0
    else:
        assert abs(got - ref) <= SIGMA_RTOL * ref, (got, ref)


def test_noalloc_sigma_of_no_element_is_zero():
    L = S.load_library()
    out = torch.full((1,), -1.0, dtype=torch.float32, device="cuda")
    st = L.smat_delta_sigma_noalloc(None, None, 0, S.SMAT_BF16, ctypes.c_float(0.1), ctypes.c_void_p(out.data_ptr()),
                                    None)
    assert st == 0
    torch.cuda.synchronize()
    assert float(out[0]) == 0.0


def test_noalloc_rejects_sizes_beyond_its_scratch_array():
    L = S.load_library()
    out = torch.empty(1, dtype=torch.float32, device="cuda")
    too_many = 16384 * 65536 + 1
    st = L.smat_delta_sigma_noalloc(ctypes.c_void_p(256), ctypes.c_void_p(512), too_many, S.SMAT_BF16,
                                    ctypes.c_float(0.1), ctypes.c_void_p(out.data_ptr()), None)
    assert st == 1  # SMAT_ERR_INVALID_ARG, before any device work
    assert b"scratch array" in L.smat_last_error()


def test_noalloc_binding_rejects_host_noncontiguous_and_bad_out():
    """The binding refuses, before calling the library, tensors the kernel
    could not read as one contiguous device array, and a result buffer that
    is not one device float."""
    th, t0 = _pair(4096, torch.bfloat16, 9)
    with pytest.raises(ValueError):
        S.delta_sigma_noalloc(th.cpu(), t0.cpu(), 0.1)
    with pytest.raises(ValueError):
        S.delta_sigma_noalloc(th[::2], t0[::2], 0.1)
    with pytest.raises(ValueError):
        S.delta_sigma_noalloc(th, t0, 0.1, out=torch.empty(1, dtype=torch.float32))
    with pytest.raises(ValueError):
        S.delta_sigma_noalloc(th, t0, 0.1, out=torch.empty(1, dtype=torch.float64, device="cuda"))
    with pytest.raises(ValueError):
        S.delta_sigma_noalloc(th, t0, 0.1, out=torch.empty(0, dtype=torch.float32, device="cuda"))
