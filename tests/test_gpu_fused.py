"""Fused statistics + forward launch: identical results with and without the
fusion, no device errors in normal runs, and the bounded wait: forward items
whose statistics are never published give up after about a second, set the
error flag (read back on the host) and leave the context usable."""

import time

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

from _parity import run_and_check_full, session_for, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def _rel_list():
    specs = [W.TensorSpec(f"t{i}", (n,), "linear" if i % 2 else "other", 0.7 if i % 2 else 1.0, 0.0, 0.1)
             for i, n in enumerate([70_001, 262_144 * 3 + 5, 17, 600_000, 4096])]
    specs.append(W.TensorSpec("fixed", (300_003,), "linear", 0.5, 1e-3, 0.0))
    return W.Workload("rel_mix", specs, O.BF16, O.BF16, 0.3, 1.0, 1, O.NOISE_GAUSSIAN, 0.02, 3e-4, seed=11)


@pytest.mark.parametrize("chunk_log2", [0, 18])
def test_fused_and_unfused_give_identical_outputs(chunk_log2):
    w = _rel_list()
    dev = torch.device("cuda")
    th, t0, sim_a, gs, go = W.generate(w, device=dev)
    sim_b = [torch.empty_like(x) for x in sim_a]
    chunk = S.SMAT_FLAG_CHUNK_LOG2(chunk_log2) if chunk_log2 else 0
    a = session_for(w, th, t0, sim_a, flags=chunk)
    b = S.SmatSession(th, t0, sim_b, [t.keep_prob for t in w.tensors], [t.sigma for t in w.tensors],
                      [t.sigma_rel for t in w.tensors], seed=w.seed, alpha_min=w.alpha_min, alpha_max=w.alpha_max,
                      alpha_mode=w.alpha_mode, noise=w.noise, flags=S.SMAT_FLAG_UNFUSED_STATS | chunk)
    for step in (0, 3):
        a.simulate_multi(step)
        b.simulate_multi(step)
        torch.cuda.synchronize()
        for x, y in zip(sim_a, sim_b):
            assert torch.equal(x.view(torch.int16), y.view(torch.int16))
    assert a.poll_errors() == 0 and b.poll_errors() == 0


@pytest.mark.parametrize("chunk_log2", [0, 18])
def test_fused_list_matches_oracle_and_reports_no_errors(chunk_log2):
    run_and_check_full(_rel_list(), steps=(0, 1, 5), flags=S.SMAT_FLAG_CHUNK_LOG2(chunk_log2) if chunk_log2 else 0)


def test_bounded_wait_runs_out_and_reports():
    w = _rel_list()
    dev = torch.device("cuda")
    th, t0, sim, gs, go = W.generate(w, device=dev)
    sess = session_for(w, th, t0, sim)
    sess.simulate_multi(0)
    assert sess.poll_errors() == 0
    # one forward item of tensor 0 (a sigma_rel tensor), its chunk 0; no statistics item publishes it
    items = torch.tensor([np.int32(np.uint32(0x80000000).view(np.int32))], dtype=torch.int32, device=dev)
    t = time.perf_counter()
    sess.debug_fused(1, items, epoch_skew=1000)
    err = sess.poll_errors()
    dt = time.perf_counter() - t
    assert err == 1, err
    assert dt < 30.0
    assert sess.poll_errors() == 0  # cleared
    # the context still works afterwards
    sess.simulate_multi(2)
    assert sess.poll_errors() == 0
    sess2 = session_for(w, th, t0, [torch.empty_like(x) for x in sim])
    sess2.simulate_multi(2)
    torch.cuda.synchronize()
    assert all(torch.equal(x.view(torch.int16), y.view(torch.int16)) for x, y in zip(sim, sess2._keep[2]))
