"""Host-side logic of runs with several ranks, on CPU with the gloo backend
(world size 2): the bench's barrier and max-over-ranks timing reduction,
per-rank experts (distinct seeds and data), and element-offset sharding of
one tensor across ranks reproducing the unsharded result bit for bit (the
oracle stands in for the per-rank compute here)."""

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out_dir):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import bench
    import oracle as O
    from paper_2609_33437_gb300 import workloads as W

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        # max over ranks of a per-rank "time"
        m = bench.max_over_ranks(1.5 + rank, world)
        # per-rank expert
        w = bench.rank_workload(W.tiny_flat(), rank)
        # one tensor sharded by element offset across the ranks
        n = 10_001
        r = np.random.default_rng(3)
        th = r.standard_normal(n).astype(np.float32)
        t0 = r.standard_normal(n).astype(np.float32)
        cut = [0, 4_096 + 17, n]
        lo, hi = cut[rank], cut[rank + 1]
        cfg = O.config(seed=5, step=2, noise=O.NOISE_GAUSSIAN, alpha_mode=O.ALPHA_PER_ELEMENT)
        part = O.simulate(cfg, O.tensor(0, hi - lo, keep_prob=0.7, sigma=1e-3, elem_offset=lo), th[lo:hi], t0[lo:hi])
        parts = [None] * world
        dist.all_gather_object(parts, (lo, part.tobytes(), w.seed, w.data_seed, m))
        if rank == 0:
            full = O.simulate(cfg, O.tensor(0, n, keep_prob=0.7, sigma=1e-3), th, t0)
            np.save(os.path.join(out_dir, "full.npy"), full)
            joined = b"".join(p[1] for p in sorted(parts, key=lambda x: x[0]))
            with open(os.path.join(out_dir, "joined.bin"), "wb") as f:
                f.write(joined)
            with open(os.path.join(out_dir, "meta.txt"), "w") as f:
                f.write(repr([(p[2], p[3], p[4]) for p in parts]))
    finally:
        dist.destroy_process_group()


def test_two_rank_host_path(tmp_path):
    port = _free_port()
    mp.start_processes(_worker, args=(2, port, str(tmp_path)), nprocs=2, join=True, start_method="spawn")
    full = np.load(tmp_path / "full.npy")
    joined = np.frombuffer((tmp_path / "joined.bin").read_bytes(), dtype=np.float32)
    assert np.array_equal(full.view(np.uint32), joined.view(np.uint32))
    meta = eval((tmp_path / "meta.txt").read_text())
    seeds = {m[0] for m in meta}
    data_seeds = {m[1] for m in meta}
    assert seeds == {0, 1} and len(data_seeds) == 2
    assert all(m[2] == 2.5 for m in meta)
