"""The bench's end-to-end leg (host buffers, copies in and out on their own
streams, the list split into pipelined groups of tensors, one session each)
returns exactly what one session over the device-resident list computes."""

import os
import sys

import pytest
import torch

from paper_2609_33437_gb300 import smat as S
from paper_2609_33437_gb300 import workloads as W

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def test_pipelined_host_io_matches_one_device_session():
    sys.path.insert(0, ROOT)
    import bench
    w = W.scaled(W.llama_7b(noise=1), 3_000_000)

    def make(th, t0, sim, idx=None):
        idx = list(range(len(w.tensors))) if idx is None else list(idx)
        ts = [w.tensors[i] for i in idx]
        return S.SmatSession(th, t0, sim, [t.keep_prob for t in ts], [t.sigma for t in ts],
                             [t.sigma_rel for t in ts], tensor_ids=idx, seed=w.seed, alpha_min=w.alpha_min,
                             alpha_max=w.alpha_max, alpha_mode=w.alpha_mode, noise=w.noise)

    hsim, hgo = bench.e2e_run(w, make, steps=2, warmup=1, world=1, groups=5, keep_outputs=True)
    th, t0, sim, gs, go = W.generate(w, device=torch.device("cuda"))
    sess = make(th, t0, sim)
    step = 1001  # the last timed step of e2e_run
    sess.simulate_multi(step)
    sess.swap()
    sess.grad_map_multi(step, gs, go)
    sess.swap()
    torch.cuda.synchronize()
    for k in range(len(w.tensors)):
        assert torch.equal(hsim[k].view(torch.int16), sim[k].cpu().view(torch.int16)), k
        assert torch.equal(hgo[k].view(torch.int16), go[k].cpu().view(torch.int16)), k
