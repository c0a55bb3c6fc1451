"""The 16-bit draw option (draw_bits = 16: every per-element draw is one
16-bit half of a Philox word, eight elements per block; keep iff the draw is
below floor(p_keep 2^16); noise from (2u + 1 - 2^16) 2^-16) through the C ABI,
element by element against the oracle with the same option: masks and
gradient maps bit-exact, uniform noise bit-exact, Gaussian and Laplace within
the tolerances of tests/_parity.py; the grid-stride, work-list, in-place and
statistics paths, both round counts, chunk and unit boundaries."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

from _parity import compare, f32_of, orc_config, orc_tensor, run_and_check_full, session_for, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    yield
    torch.cuda.synchronize()


def _ragged(dtype, alpha_mode, noise, rel=False, seed=0x16B1_7D2A):
    sizes = [0, 1, 7, 8, 9, 15, 16, 17, 33, 131_073, 262_144, 262_153, 600_003]
    keeps = [0.5, 0.9, 0.1, 0.7, 1.0, 0.0, 0.3, 0.5, 0.7, 0.9, 0.3, 0.5 + 2**-10, 0.7]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 0.0 if rel and i % 3 == 0 else (2e-3 if i % 4 else 0.0),
                          0.1 if rel and i % 3 == 0 else 0.0) for i, n in enumerate(sizes)]
    return W.Workload(f"d16_{dtype}_{alpha_mode}_{noise}_{rel}", specs, dtype, dtype, 0.2, 1.0, alpha_mode, noise,
                      0.02, 1e-3, seed=seed)


@pytest.mark.parametrize("noise", [O.NOISE_UNIFORM, O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
@pytest.mark.parametrize("alpha_mode", [O.ALPHA_GLOBAL, O.ALPHA_PER_TENSOR, O.ALPHA_PER_ELEMENT])
@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_draw16_modes_small_ragged_list(dtype, alpha_mode, noise):
    run_and_check_full(_ragged(dtype, alpha_mode, noise), steps=(0, 7), draw_bits=16)


@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_draw16_sigma_rel_work_list_and_unfused(dtype):
    """sigma_rel tensors: the statistics ride in the work-list launch (and, with
    SMAT_FLAG_UNFUSED_STATS, run as their own pass before a grid-stride
    forward); same results either way."""
    w = _ragged(dtype, O.ALPHA_PER_TENSOR, O.NOISE_GAUSSIAN, rel=True)
    run_and_check_full(w, steps=(0, 3), draw_bits=16)
    run_and_check_full(w, steps=(1,), draw_bits=16, flags=S.SMAT_FLAG_UNFUSED_STATS)


@pytest.mark.parametrize("chunk_log2", [12, 18])
def test_draw16_seven_rounds_accumulate_f32_grads_and_chunks(chunk_log2):
    specs = [W.TensorSpec("a", (70_001,), "linear", 0.7, 1e-3), W.TensorSpec("b", (9,), "other", 1.0, 1e-3),
             W.TensorSpec("c", (262_144 + 40,), "linear", 0.3, 1e-3)]
    w = W.Workload("d16_r7", specs, O.BF16, O.BF16, 0.3, 1.0, O.ALPHA_PER_ELEMENT, O.NOISE_GAUSSIAN, 0.02, 1e-3,
                   seed=51)
    run_and_check_full(w, steps=(1,), rounds=7, accumulate=True, gdtype=O.F32, draw_bits=16,
                       flags=S.SMAT_FLAG_CHUNK_LOG2(chunk_log2))


def test_draw16_element_offsets_and_in_place_gradient():
    """Shards at element offsets (odd, not a multiple of 8, and above 2^35,
    where the block index needs counter word 1) take the element path or the
    vector path and still equal the oracle; the gradient map in place."""
    dev = torch.device("cuda")
    n = 50_000
    specs = [W.TensorSpec("a", (n,), "linear", 0.7, 2e-3)] * 3
    w = W.Workload("d16_off", specs, O.BF16, O.BF16, 0.3, 1.0, O.ALPHA_PER_ELEMENT, O.NOISE_GAUSSIAN, 0.02, 1e-3,
                   seed=77)
    th, t0, sim, gs, go = W.generate(w, device=dev)
    offs = [3, 16 * 1001, (5 << 35) + 16]
    sess = session_for(w, th, t0, sim, elem_offsets=offs, draw_bits=16)
    g_in = [g.clone() for g in gs]
    hgs = [to_host(g) for g in gs]
    sess.simulate_multi(4)
    sess.swap()
    sess.grad_map_multi(4, g_in, g_in)  # g_out == g_sim
    sess.swap()
    torch.cuda.synchronize()
    cfg = orc_config(w, 4, draw_bits=16)
    for k in range(3):
        t = orc_tensor(w, k, elem_offset=offs[k])
        ref = O.simulate(cfg, t, to_host(th[k]), to_host(t0[k]))
        compare(to_host(sim[k]), ref.view(np.uint16), O.BF16, O.NOISE_GAUSSIAN, f32_of(to_host(th[k])),
                f32_of(to_host(t0[k])), what=f"offset {offs[k]}")
        gref = O.gradmap(cfg, t, hgs[k], gdtype=O.BF16)
        assert np.array_equal(to_host(g_in[k]).view(np.uint16), gref.view(np.uint16)), k
        bits = sess.mask_bits(4, k).cpu().numpy().view(np.uint32)
        assert np.array_equal(bits, O.mask_bits(cfg, t)), k
    assert sess.poll_errors() == 0
    sess.close()


@pytest.mark.parametrize("noise", [O.NOISE_GAUSSIAN, O.NOISE_LAPLACE])
@pytest.mark.parametrize("dtype", [O.BF16, O.F32])
def test_draw16_in_place_theta0(dtype, noise):
    """In-place mode (the sim buffer holds theta0 and is overwritten with
    theta~; flagged groups are recomputed whole) with 16-bit draws."""
    sizes = [70_001, 262_144 * 2 + 48, 17, 4096, 300_003]
    keeps = [0.7, 0.5 + 2**-10, 0.9, 1.0, 0.3]
    specs = [W.TensorSpec(f"t{i}", (n,), "linear", keeps[i], 2e-3) for i, n in enumerate(sizes)]
    w = W.Workload(f"d16_ip_{dtype}_{noise}", specs, dtype, dtype, 0.3, 1.0, O.ALPHA_PER_TENSOR, noise, 0.02, 1e-3,
                   seed=0xD16)
    th, t0, sim, gs, go = W.generate(w, device=torch.device("cuda"))
    buf = [x.clone() for x in t0]
    ip = session_for(w, th, buf, buf, draw_bits=16)
    ip.simulate_multi(2)
    torch.cuda.synchronize()
    cfg = orc_config(w, 2, draw_bits=16)
    for k in range(len(sizes)):
        ref = O.simulate(cfg, orc_tensor(w, k), to_host(th[k]), to_host(t0[k]))
        compare(to_host(buf[k]), ref.view(np.uint16 if dtype == O.BF16 else np.uint32), dtype, noise,
                f32_of(to_host(th[k])), f32_of(to_host(t0[k])), what=f"in-place tensor {k}")
    assert ip.poll_errors() == 0
    ip.close()


def test_draw16_larger_bf16_list():
    """A 0.5B-style list cut to about 2e7 elements (bf16, fp32 gradients):
    every element against the oracle, one step."""
    w = W.scaled(W.dec_0p5b(), 20_000_000)
    run_and_check_full(w, steps=(5,), draw_bits=16)
