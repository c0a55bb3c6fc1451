#!/usr/bin/env python
"""Benchmark of the SMAT simulated-merge hot path on GB300.

One step = one SMAT simulated-loss step's worth of the hot path over the
whole parameter list: delta statistics (sigma_t = 0.1 std(delta) per tensor),
per-call scalars, the fused forward theta~ = theta0 + alpha m (.) (theta -
theta0) + eps, the storage swap, the gradient map g = alpha m (.) g~ and the
swap back. Workload: the 7B Llama-style list in bf16 (291 tensors,
6,738,415,616 elements, bf16 gradients), Gaussian eps, per-tensor alpha ~
U[0.3, 1), p_keep 0.7 on attention/MLP linears.

Metric: algorithmic HBM bytes of the step / step time (GB/s), plus params/s.
Algorithmic bytes per element: 2b (statistics: theta, theta0) + 3b (forward:
theta, theta0 in, theta~ out) + 2gb (gradient: g~ in, g out) = 14 B in bf16.

N > 1 (torchrun): each rank runs its own expert's full list (independent
problems, weak scaling, no collective on the data path); value is the bytes
of all ranks over the slowest rank's time.

--impl reference runs the CPU oracle (the reference arm of this benchmark)
on a bounded sample of the same workload, on the host cores, rank 0 only.

--sweep PATH measures the flat-tensor sweep instead (one tensor of n = 2^16
.. 2^32 elements, fp32 and bf16, p_keep 0.1 .. 0.9, alpha per tensor or per
element ~ U[0, 1), sigma 0 or 1e-4 Gaussian): forward alone and forward +
gradient map, median of 20 CUDA-event-timed repetitions after 3 warm-ups,
L2 flushed before each; one JSON line per point to PATH and a summary line
on stdout.
"""

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2609_33437_gb300 import workloads as W  # noqa: E402

METRIC = "simulated-merge fwd+grad-map HBM GB/s (fraction of GB300 peak); params/sec"
UNIT = "GB/s"
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0
KERNEL_SOURCES = [os.path.join(ROOT, "paper_2609_33437_gb300", "csrc", f)
                  for f in ("smat_device.cuh", "smat_simulate.cuh", "smat_fused_bf16.cu", "smat_gradmap.cu",
                            "smat_internal.h")]


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["smat", "reference"], default="smat")
    ap.add_argument("--workload", default="llama_7b", choices=["llama_7b", "dec_0p5b", "vl_7b", "tiny_flat"])
    ap.add_argument("--noise", choices=["gaussian", "uniform", "laplace"], default="gaussian")
    ap.add_argument("--scale", type=int, default=0, help="cut the list to about this many elements (profiling)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--theta0", choices=["device", "inplace", "host"], default="device",
                    help="where theta0 lives: its own HBM buffer (default); in-place (the sim buffer holds theta0 "
                         "and is refilled from pinned host memory every step, inside the timed region); pinned "
                         "host memory read directly by the kernels")
    ap.add_argument("--chunk-log2", type=int, default=0,
                    help="force the work-chunk size to 2^k elements (12..18; 0: the per-list rule)")
    ap.add_argument("--philox-rounds", type=int, choices=[7, 10], default=10,
                    help="Philox-4x32 rounds of the random streams (10 is the default stream definition)")
    ap.add_argument("--draw-bits", type=int, choices=[32, 16], default=32,
                    help="per-element draw width: 32 (the default stream definition) or 16 (the 16-bit draw "
                         "option: eight elements per Philox block, no mask-tie path; a different stream)")
    ap.add_argument("--sweep", metavar="PATH", default=None,
                    help="run the flat-tensor sweep, one JSON line per point to PATH")
    ap.add_argument("--sweep-max-log2n", type=int, default=32)
    ap.add_argument("--sweep-min-log2n", type=int, default=16)
    ap.add_argument("--merge", choices=["wa", "ta", "dare", "ties"], default=None,
                    help="time merging K experts of the chosen list (Eq. merged-state) instead of the SMAT step")
    ap.add_argument("--experts", type=int, default=8)
    ap.add_argument("--ref-sample", type=int, default=0,
                    help="elements per step of the oracle sample in --impl reference (0: sized for about 150 s)")
    ap.add_argument("--adamw", action="store_true",
                    help="time the gradient map fused with an AdamW step on the chosen list, beside the plain map")
    ap.add_argument("--schedule", action="store_true",
                    help="training-loop overhead of periodic SMAT (Sec. 4.3) over plain fine-tuning, synthetic model")
    return ap.parse_args()


NOISE_CODE = {"uniform": 0, "gaussian": 1, "laplace": 2}
NOISE_NAME = {v: k for k, v in NOISE_CODE.items()}


def workload(args) -> W.Workload:
    if args.workload == "llama_7b":
        w = W.llama_7b(noise=NOISE_CODE[args.noise])
    else:
        w = W.WORKLOADS[args.workload]()
        if args.noise != "gaussian":
            w.noise = NOISE_CODE[args.noise]
    if args.scale:
        w = W.scaled(w, args.scale)
    return w


def step_bytes(w: W.Workload) -> dict:
    b = 2 if w.dtype == W.BF16 else 4
    gb = 2 if w.gdtype == W.BF16 else 4
    n_rel = sum(t.numel for t in w.tensors if t.sigma_rel > 0)
    return {"delta_stats": 2 * b * n_rel, "simulate": 3 * b * w.numel, "gradmap": 2 * gb * w.numel}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_hash():
    import hashlib
    h = hashlib.sha256()
    for p in KERNEL_SOURCES:
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, wname: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel source (else None)."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(p) as f:
            d = json.load(f)
        rec = d.get(kernel, {}).get(wname)
        if rec and rec.get("kernel_hash") == kernel_hash():
            return rec
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.samples = []
        self.proc = None
        self.marks = []
        try:
            uuid = "GPU-" + str(torch.cuda.get_device_properties(device_index).uuid)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", uuid, f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.perf_counter(), line.strip()))

    def mark(self):
        self.marks.append(time.perf_counter())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        t0, t1 = (self.marks + [0, 0])[:2]
        rows = [s for t, s in self.samples if t0 <= t <= t1 + 0.15] or [s for _, s in self.samples[-3:]]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            f = [x.strip() for x in r.split(",")]
            if len(f) < 8:
                continue
            try:
                sm.append(float(f[0]))
                mx.append(float(f[1]))
            except ValueError:
                continue
            for name, v in zip(names, f[4:8]):
                if v.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    """Slowest rank's value (NCCL on the GPU, gloo on the host)."""
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def rank_workload(w: W.Workload, rank: int) -> W.Workload:
    """Rank r trains its own expert: its own SMAT seed and its own data."""
    w.seed = rank
    w.data_seed = w.data_seed + 1000 * rank
    return w


# ------------------------------------------------------------ CPU oracle ---

def oracle_run(w: W.Workload, max_elems: int, step: int = 0, threads: int = 1):
    """Oracle forward + gradient map over a sample of w: every tensor of w
    scaled so the sample totals about max_elems (all shapes and settings
    kept). The inputs are generated first (untimed); with threads > 1 the
    tensors are handed to that many threads (the oracle keeps no shared
    state, and its calls run without the interpreter lock). Returns
    (seconds, algorithmic bytes, elements, sample name)."""
    import concurrent.futures as cf
    import oracle as O
    s = W.scaled(w, max_elems)
    gen = torch.Generator().manual_seed(99)
    cfg = O.config(seed=w.seed, step=step, alpha_mode=w.alpha_mode, noise=w.noise, alpha_min=w.alpha_min,
                   alpha_max=w.alpha_max)

    def host(x, dt):
        x = x.to(W.torch_dtype(dt))
        return x.view(torch.int16).numpy().view(np.uint16) if dt == W.BF16 else x.numpy()

    items = []
    for k, spec in enumerate(s.tensors):
        n = spec.numel
        t0f = torch.randn(n, generator=gen) * w.theta0_std
        thf = t0f + torch.randn(n, generator=gen) * w.delta_std
        gf = torch.randn(n, generator=gen)
        t = O.tensor(k, n, dtype=w.dtype, keep_prob=spec.keep_prob, sigma=spec.sigma, sigma_rel=spec.sigma_rel)
        items.append((t, host(thf, w.dtype), host(t0f, w.dtype), host(gf, w.gdtype)))

    def one(item):
        t, th, t0, g = item
        O.simulate(cfg, t, th, t0)
        O.gradmap(cfg, t, g, gdtype=w.gdtype)

    a = time.perf_counter()
    if threads > 1:
        # largest tensors first, so the threads end together
        order = sorted(items, key=lambda it: -it[0].numel)
        with cf.ThreadPoolExecutor(max_workers=threads) as ex:
            list(ex.map(one, order))
    else:
        for it in items:
            one(it)
    secs = time.perf_counter() - a
    nbytes = sum(step_bytes(s).values())
    return secs, nbytes, s.numel, f"{s.name}: {len(s.tensors)} tensors, {s.numel} elements"


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    w = workload(args)
    # about 150 s in all: the oracle takes about 1 us per element (forward +
    # gradient map on one Grace core) plus the sample's input generation
    per_step = int(min(8_000_000, max(200_000, 150.0 / max(1, args.steps + args.warmup) / 1.1e-6)))
    if args.ref_sample > 0:
        per_step = args.ref_sample
    for _ in range(args.warmup):
        oracle_run(w, per_step)
    tot_s, tot_b, tot_n = 0.0, 0, 0
    sample = ""
    for _ in range(args.steps):
        s, b, n, sample = oracle_run(w, per_step)
        tot_s += s
        tot_b += b
        tot_n += n
    value = tot_b / tot_s / 1e9
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / args.steps,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
           "data": "synthetic", "params_per_s": tot_n / tot_s,
           "config": {"workload": w.name, "elements_per_step_sample": tot_n // args.steps,
                      "noise": NOISE_NAME[w.noise]},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                            "sample": f"each step: {sample} (single-threaded C++ oracle, forward + gradient map)"},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out))
    return 0


# ------------------------------------------------------------- GPU path ---

def host_available_bytes():
    try:
        return os.sysconf("SC_AVPHYS_PAGES") * os.sysconf("SC_PAGE_SIZE")
    except Exception:
        return 0


def gpu_local_cpus(device_index: int):
    """CPUs of the NUMA node the GPU's PCI function reports (sysfs), or None."""
    try:
        p = torch.cuda.get_device_properties(device_index)
        dev = "%04x:%02x:%02x.0" % (p.pci_domain_id, p.pci_bus_id, p.pci_device_id)
        with open(f"/sys/bus/pci/devices/{dev}/numa_node") as f:
            node = int(f.read().strip())
        if node < 0:
            return None
        with open(f"/sys/devices/system/node/node{node}/cpulist") as f:
            spec = f.read().strip()
        cpus = set()
        for part in spec.split(","):
            if part:
                a, _, b = part.partition("-")
                cpus.update(range(int(a), int(b or a) + 1))
        return (node, cpus) if cpus else None
    except Exception:
        return None


HUGE_PAGE = 512 << 20  # transparent huge page size of an arm64 kernel with 64 KB base pages


class PinnedHost:
    """Pinned host buffers for the end-to-end leg. Each one is an anonymous
    mapping advised for transparent huge pages (madvise(MADV_HUGEPAGE)),
    faulted in and registered with cudaHostRegister: the copy engines then
    translate a few hundred large pages instead of about a million 64 KB ones
    (measured: a step's 67 GB of copies at about 240 GB/s instead of 165 when
    the kernel had huge pages free; where it has none the mapping keeps base
    pages, see huge_page_fraction()). Falls back to torch's pinned allocator
    where any step fails. close() unregisters them."""

    def __init__(self):
        self._maps, self._registered = [], []
        self.huge = True

    def empty(self, n, dtype):
        import ctypes
        import mmap
        nbytes = n * torch.empty((), dtype=dtype).element_size()
        if self.huge and nbytes > 0:
            try:
                m = mmap.mmap(-1, nbytes + HUGE_PAGE, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
                m.madvise(mmap.MADV_HUGEPAGE)
                base = ctypes.addressof(ctypes.c_char.from_buffer(m))
                raw = torch.frombuffer(m, dtype=torch.uint8, count=nbytes, offset=(-base) % HUGE_PAGE)
                raw.fill_(0)  # fault the pages in (huge pages where the kernel has them)
                if int(torch.cuda.cudart().cudaHostRegister(raw.data_ptr(), nbytes, 0)) == 0:
                    self._maps.append(m)
                    self._registered.append(raw)
                    return raw.view(dtype)
                del raw
                m.close()
            except Exception:
                pass
            self.huge = False
        return torch.empty(n, dtype=dtype, pin_memory=True)

    def huge_page_fraction(self):
        """Share of this process's anonymous memory backed by transparent huge
        pages (AnonHugePages / Anonymous in /proc/self/smaps_rollup), or None:
        where the kernel had no free huge pages the buffers fall back to base
        pages and the copies slow down."""
        try:
            vals = {}
            with open("/proc/self/smaps_rollup") as f:
                for line in f:
                    k, _, rest = line.partition(":")
                    if k in ("AnonHugePages", "Anonymous"):
                        vals[k] = int(rest.split()[0])
            return vals["AnonHugePages"] / vals["Anonymous"] if vals.get("Anonymous") else None
        except Exception:
            return None

    def numa_pages(self):
        """Pages of this process's anonymous mappings per NUMA node (summed
        N<node>=<pages> fields of /proc/self/numa_maps), or None: host buffers
        that did not fit on the GPU's node land on another one, behind a
        slower path."""
        try:
            nodes = {}
            with open("/proc/self/numa_maps") as f:
                for line in f:
                    if "anon" not in line:
                        continue
                    kb = 4
                    for tok in line.split():
                        if tok.startswith("kernelpagesize_kB="):
                            kb = int(tok.split("=")[1])
                    for tok in line.split():
                        if tok.startswith("N") and "=" in tok and tok[1:tok.index("=")].isdigit():
                            node = tok[1:tok.index("=")]
                            nodes[node] = nodes.get(node, 0) + int(tok.split("=")[1]) * kb * 1024
            return {k: v for k, v in sorted(nodes.items())} or None
        except Exception:
            return None

    def close(self):
        for raw in self._registered:
            torch.cuda.cudart().cudaHostUnregister(raw.data_ptr())
        self._registered.clear()
        self._maps.clear()


def step_copy_roof(h_ins, h_outs, d_ins, d_outs, groups=8, reps=2):
    """The end-to-end step's copies alone, in the pipeline's pattern: the
    arrays cut into `groups` consecutive ranges; for each range every input
    array is copied in on one stream while the output arrays are copied out
    on another, no kernels (the roof of the end-to-end leg on this machine's link
    and these host buffers). Returns GB/s of host traffic."""
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    nbytes = sum(h.numel() * h.element_size() for h in h_ins + h_outs)
    n = h_ins[0].numel()
    per = (n + groups - 1) // groups
    best = float("inf")
    for _ in range(reps):
        torch.cuda.synchronize()
        t = time.perf_counter()
        for g in range(groups):
            a, b = g * per, min(n, (g + 1) * per)
            with torch.cuda.stream(s1):
                for h, d in zip(h_ins, d_ins):
                    d[a:b].copy_(h[a:b], non_blocking=True)
            with torch.cuda.stream(s2):
                for h, d in zip(h_outs, d_outs):
                    h[a:b].copy_(d[a:b], non_blocking=True)
        torch.cuda.synchronize()
        best = min(best, time.perf_counter() - t)
    return nbytes / best / 1e9


def link_roof(h_in, h_out, nbytes=4 << 30, reps=3, max_streams=4):
    """Host-link copy roof on this machine: pinned-host-to-device and
    device-to-pinned-host cudaMemcpyAsync (torch copy_, non_blocking) of
    `nbytes` in each direction, split over 1, 2 or 4 streams at once (several
    copy engines), alone and both directions together; best of `reps` for each,
    timed with CUDA events. h_in / h_out: pinned host tensors of at least
    nbytes. Returns the best rate of each kind and the rates per stream count."""
    hi = h_in.view(-1).view(torch.uint8)
    ho = h_out.view(-1).view(torch.uint8)
    nbytes = min(nbytes, hi.numel(), ho.numel())
    hi, ho = hi[:nbytes], ho[:nbytes]
    d1 = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    d2 = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    streams = [torch.cuda.Stream() for _ in range(2 * max_streams)]

    def timed(which, k):
        best = float("inf")
        parts = [(p * nbytes // k, (p + 1) * nbytes // k) for p in range(k)]
        for _ in range(reps):
            torch.cuda.synchronize()
            e0 = torch.cuda.Event(enable_timing=True)
            e0.record(streams[0])
            ends = []
            for p, (a, b) in enumerate(parts):
                for d, (src, dst) in enumerate(((hi, d1), (d2, ho))):
                    if (which == "h2d" and d == 1) or (which == "d2h" and d == 0):
                        continue
                    st = streams[2 * p + d]
                    st.wait_event(e0)
                    with torch.cuda.stream(st):
                        dst[a:b].copy_(src[a:b], non_blocking=True)
                    e = torch.cuda.Event(enable_timing=True)
                    e.record(st)
                    ends.append(e)
            torch.cuda.synchronize()
            best = min(best, max(e0.elapsed_time(e) for e in ends) / 1e3)
        return best

    out = {"bytes_per_direction": nbytes, "per_streams": {}}
    for k in (1, 2, max_streams):
        r = {"h2d": nbytes / timed("h2d", k) / 1e9, "d2h": nbytes / timed("d2h", k) / 1e9,
             "bidirectional": 2 * nbytes / timed("both", k) / 1e9}
        out["per_streams"][k] = r
    for kind in ("h2d", "d2h", "bidirectional"):
        out[kind] = max(r[kind] for r in out["per_streams"].values())
    del d1, d2
    return out


def e2e_run(w, sess_factory, steps, warmup, world, groups=8, keep_outputs=False, copy_streams=2):
    """The same step through the public API with host inputs: pinned host
    theta, theta0 and g~ are copied in and theta~ and g copied out every
    step, inside the timed region. The list is cut into `groups` groups of
    consecutive tensors (one session each, same tensor ids, so the results
    are those of one session). A group's tensors are views of one device
    buffer per array, laid out as on the host (a tensor whose size is not a
    multiple of 16 elements pads the next one's start to keep 32-byte
    alignment), so a group moves with a few large copies, each split over
    `copy_streams` streams per direction so several copy engines work at once.
    Groups and steps are pipelined: group k's inputs of step s + 1 are copied
    in as soon as its compute of step s has read them, its results copied out
    while later groups compute; the timed region ends when the results of the
    last step are on the host."""
    dev = torch.device("cuda")
    tdt, gdt = W.torch_dtype(w.dtype), W.torch_dtype(w.gdtype)
    n = w.numel
    nt = len(w.tensors)
    # host buffers and copies on the CPUs next to the GPU (first-touch placement)
    local = gpu_local_cpus(torch.cuda.current_device())
    saved = os.sched_getaffinity(0) if local else None
    if local:
        os.sched_setaffinity(0, local[1])
    pinned = PinnedHost()
    h_th = pinned.empty(n, tdt)
    h_t0 = pinned.empty(n, tdt)
    h_gs = pinned.empty(n, gdt)
    h_sim = pinned.empty(n, tdt)
    h_go = pinned.empty(n, gdt)
    offs = np.cumsum([0] + [t.numel for t in w.tensors])
    # groups of consecutive tensors with about n / groups elements each
    cuts, target, acc, start = [], n / max(1, groups), 0, 0
    for k, t in enumerate(w.tensors):
        acc += t.numel
        if acc >= target * (len(cuts) + 1) or k == nt - 1:
            cuts.append(list(range(start, k + 1)))
            start = k + 1
    # per group: device offsets of its tensors (16-element aligned) and the
    # runs of tensors whose device layout equals the host layout
    bufs, views, runs = [], [None] * nt, []
    for ks in cuts:
        doff, d = {}, 0
        for k in ks:
            d = (d + 15) // 16 * 16
            doff[k] = d
            d += w.tensors[k].numel
        gb = {name: torch.empty(max(d, 1), dtype=(gdt if name in ("gs", "go") else tdt), device=dev)
              for name in ("th", "t0", "gs", "sim", "go")}
        bufs.append(gb)
        for k in ks:
            a, b = doff[k], doff[k] + w.tensors[k].numel
            views[k] = {name: buf[a:b] for name, buf in gb.items()}
        r = []
        for k in ks:
            if r and doff[k] - int(offs[k]) == r[-1][2]:
                r[-1][1] = int(offs[k + 1])
            else:
                r.append([int(offs[k]), int(offs[k + 1]), doff[k] - int(offs[k])])
        runs.append(r)
    for k in range(nt):
        th, t0, g = W.generate_tensor(w, k, dev)
        a, b = int(offs[k]), int(offs[k + 1])
        h_th[a:b].copy_(th)
        h_t0[a:b].copy_(t0)
        h_gs[a:b].copy_(g)
        views[k]["th"].copy_(th)
        views[k]["t0"].copy_(t0)
        views[k]["gs"].copy_(g)
        del th, t0, g
    sessions = [sess_factory([views[k]["th"] for k in ks], [views[k]["t0"] for k in ks],
                             [views[k]["sim"] for k in ks], ks) for ks in cuts]
    s_in = [torch.cuda.Stream() for _ in range(copy_streams)]
    s_out = [torch.cuda.Stream() for _ in range(copy_streams)]
    s_cmp = torch.cuda.Stream()
    done = [None] * len(cuts)    # compute of the group finished (its inputs are free)
    copied = [None] * len(cuts)  # results of the group copied out (its outputs are free)

    def pieces(a, b):
        # split [a, b) into copy_streams parts when it is large enough to gain from it
        if b - a < (32 << 20):
            return [(0, a, b)]
        return [(p, a + p * (b - a) // copy_streams, a + (p + 1) * (b - a) // copy_streams)
                for p in range(copy_streams)]

    def one(step):
        for gi, ks in enumerate(cuts):
            gb = bufs[gi]
            ev_in = []
            for p, st in enumerate(s_in):
                if done[gi] is not None:
                    st.wait_event(done[gi])
            for a0, b0, shift in runs[gi]:
                for p, a, b in pieces(a0, b0):
                    with torch.cuda.stream(s_in[p]):
                        gb["th"][a + shift:b + shift].copy_(h_th[a:b], non_blocking=True)
                        gb["t0"][a + shift:b + shift].copy_(h_t0[a:b], non_blocking=True)
                        gb["gs"][a + shift:b + shift].copy_(h_gs[a:b], non_blocking=True)
            for st in s_in:
                e = torch.cuda.Event()
                e.record(st)
                s_cmp.wait_event(e)
            if copied[gi] is not None:
                for e in copied[gi]:
                    s_cmp.wait_event(e)
            sess = sessions[gi]
            sess.simulate_multi(step, stream=s_cmp)
            sess.swap()
            sess.grad_map_multi(step, [views[k]["gs"] for k in ks], [views[k]["go"] for k in ks], stream=s_cmp)
            sess.swap()
            done[gi] = torch.cuda.Event()
            done[gi].record(s_cmp)
            for st in s_out:
                st.wait_event(done[gi])
            for a0, b0, shift in runs[gi]:
                for p, a, b in pieces(a0, b0):
                    with torch.cuda.stream(s_out[p]):
                        h_sim[a:b].copy_(gb["sim"][a + shift:b + shift], non_blocking=True)
                        h_go[a:b].copy_(gb["go"][a + shift:b + shift], non_blocking=True)
            copied[gi] = []
            for st in s_out:
                e = torch.cuda.Event()
                e.record(st)
                copied[gi].append(e)

    for s in range(warmup):
        one(s)
    torch.cuda.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    a = time.perf_counter()
    for s in range(steps):
        one(1000 + s)
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - a, world)
    bytes_step = sum(step_bytes(w).values())
    h2d = 2 * h_th.element_size() * n + h_gs.element_size() * n
    d2h = h_sim.element_size() * n + h_go.element_size() * n
    for sess in sessions:
        sess.close()
    if keep_outputs:  # the last step's theta~ and g on the host (tests)
        if saved:
            os.sched_setaffinity(0, saved)
        hv = lambda h: [h[int(offs[k]):int(offs[k + 1])].clone() for k in range(nt)]  # noqa: E731
        out = hv(h_sim), hv(h_go)
        pinned.close()
        return out
    del bufs, views
    torch.cuda.empty_cache()
    roof = link_roof(h_th, h_sim)
    d_in = [torch.empty_like(h, device=dev) for h in (h_th, h_t0, h_gs)]
    d_out = [torch.empty_like(h, device=dev) for h in (h_sim, h_go)]
    roof["step_copies"] = step_copy_roof([h_th, h_t0, h_gs], [h_sim, h_go], d_in, d_out)
    del d_in, d_out
    if saved:
        os.sched_setaffinity(0, saved)
    huge = pinned.huge
    huge_frac = pinned.huge_page_fraction() if huge else None
    numa = pinned.numa_pages()
    pinned.close()
    host_gbs = (h2d + d2h) * steps / el / 1e9
    return {"value": world * bytes_step * steps / el / 1e9, "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "ms_per_step": 1e3 * el / steps, "workload": w.name,
            "pipeline": f"{len(cuts)} tensor groups, steps and groups pipelined over {copy_streams} copy-in, "
                        f"one compute and {copy_streams} copy-out streams",
            "host_numa_node": local[0] if local else None,
            "host_buffers": "huge-page mappings registered with cudaHostRegister" if huge else "torch pinned memory",
            "host_huge_page_fraction": huge_frac,
            "host_bytes_per_numa_node": numa,
            "host_link_gbs": host_gbs, "link_roof_gbs": roof,
            "frac_of_link_roof": host_gbs / roof["step_copies"] if roof["step_copies"] > 0 else None}


def run_smat(args):
    world, rank, local = dist_setup(args)
    from paper_2609_33437_gb300 import smat as S
    S.load_library()
    dev = torch.device("cuda", local)
    w = rank_workload(workload(args), rank)

    def make_session(th, t0, sim, idx=None):
        # idx: the tensors' positions in the list (their ids; all tensors by default)
        idx = list(range(len(w.tensors))) if idx is None else list(idx)
        ts = [w.tensors[i] for i in idx]
        return S.SmatSession(th, t0, sim, [t.keep_prob for t in ts], [t.sigma for t in ts],
                             [t.sigma_rel for t in ts], tensor_ids=idx, seed=w.seed, alpha_min=w.alpha_min,
                             alpha_max=w.alpha_max, alpha_mode=w.alpha_mode, noise=w.noise,
                             philox_rounds=args.philox_rounds, draw_bits=args.draw_bits,
                             flags=S.SMAT_FLAG_CHUNK_LOG2(args.chunk_log2) if args.chunk_log2 else 0)

    th, t0, sim, gs, go = W.generate(w, device=dev)
    host_t0 = None
    pinned = None
    if args.theta0 in ("host", "inplace"):
        # theta0 in pinned host memory: one huge-page mapping registered with
        # cudaHostRegister (see PinnedHost), one view per tensor
        pinned = PinnedHost()
        pad = lambda n: (n + 15) // 16 * 16  # noqa: E731  (32-byte aligned views: the vector path)
        flat = pinned.empty(sum(pad(x.numel()) for x in t0), t0[0].dtype if t0 else torch.bfloat16)
        views, off = [], 0
        for x in t0:
            v = flat[off:off + x.numel()].view(x.shape)
            v.copy_(x)
            views.append(v)
            off += pad(x.numel())
        if args.theta0 == "host":
            t0 = views
        else:
            host_t0 = views
            sim = t0  # one buffer per tensor: theta0, overwritten by theta~, refilled every step
    sess = make_session(th, t0, sim)

    def step(s):
        sess.simulate_multi(s)
        sess.swap()
        sess.grad_map_multi(s, gs, go)
        sess.swap()
        if host_t0 is not None:
            sess.refill_theta0(host_t0)

    for s in range(args.warmup):
        step(s)
    torch.cuda.synchronize()
    clocks = None if args.no_clocks else ClockSampler(local)
    if clocks:
        time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize()
    sess.timing_enable(True)
    stream = torch.cuda.current_stream()
    # lists whose step moves less than 1 GB could be served from the 129 MB L2
    # across steps: write 256 MB before each step and time the steps one by one
    small = sum(step_bytes(w).values()) < (1 << 30)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev) if small else None
    if clocks:
        clocks.mark()
    if small:
        ms = 0.0
        for s in range(args.steps):
            flush.zero_()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            step(100 + s)
            e1.record(stream)
            e1.synchronize()
            ms += e0.elapsed_time(e1)
    else:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(args.steps):
            step(100 + s)
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1)
    if clocks:
        clocks.mark()
    barrier(world)
    kern = sess.timing_read()
    sess.timing_enable(False)
    clk = clocks.stop() if clocks else None
    ms_step = max_over_ranks(ms / args.steps, world)

    nb = step_bytes(w)
    bytes_step = sum(nb.values())
    fused = kern["delta_stats"][1] == 0 and nb["delta_stats"] > 0
    if fused:  # statistics run inside the forward launch
        nb = dict(nb, simulate=nb["simulate"] + nb["delta_stats"], delta_stats=0)
    value = world * bytes_step / (ms_step * 1e-3) / 1e9
    peak, peak_kind = measured_peaks()
    sim_ms, sim_n = kern["simulate"]
    sim_avg = sim_ms / max(1, sim_n)
    achieved = nb["simulate"] / (sim_avg * 1e-3) / 1e9
    traffic = recorded_traffic("simulate", w.name)
    per_kernel = {}
    for k, (kms, kn) in kern.items():
        if kn == 0:
            continue
        per_kernel[k] = {"avg_ms": kms / kn, "launches": kn, "share": kms / max(1e-9, sum(v[0] for v in kern.values()))}
        if k in nb and nb[k]:
            per_kernel[k]["gbs"] = nb[k] / (kms / kn * 1e-3) / 1e9
            per_kernel[k]["frac_of_measured_peak"] = per_kernel[k]["gbs"] / peak
    launches = int(sum(v[1] for v in kern.values()))
    del sess
    if pinned is not None:
        del t0, host_t0, views, flat
        pinned.close()
    out = None
    if rank == 0:
        out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
               "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
               "vs_baseline": None, "dtype": "bf16" if w.dtype == W.BF16 else "f32",
               "data": "synthetic (seeded torch draws shaped like a 7B Llama-style parameter list)",
               "params_per_s": world * w.numel / (ms_step * 1e-3),
               "frac_of_measured_peak": value / peak, "frac_of_nominal_8tbs": value / NOMINAL_HBM_GBS,
               "config": {"workload": w.name, "tensors": len(w.tensors), "elements": w.numel,
                          "param_dtype": "bf16" if w.dtype == W.BF16 else "f32",
                          "grad_dtype": "bf16" if w.gdtype == W.BF16 else "f32",
                          "noise": NOISE_NAME[w.noise], "alpha": f"per-tensor U[{w.alpha_min}, {w.alpha_max})",
                          "philox_rounds": args.philox_rounds, "draw_bits": args.draw_bits,
                          "bytes_per_step": bytes_step,
                          "l2": ("256 MB written before each timed step (the step's data would fit in L2)" if small
                                 else "inputs larger than L2 (no flush needed)"),
                          "theta0": args.theta0,
                          "parallelism": f"{world} independent experts (one per GPU)"},
               "kernels": per_kernel,
               "roofline": {"bound": "hbm", "kernel": "stats_simulate (fused)" if fused else "simulate",
                            "achieved": achieved, "peak": peak,
                            "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                            "traffic": traffic["dram_bytes_per_launch"] if traffic else None,
                            "algorithmic_bytes_per_launch": nb["simulate"]},
               "clocks": clk, "gpu_launches": launches}
    if out is not None and args.theta0 != "device":
        kern_ms = sum(v["avg_ms"] * v["launches"] for v in per_kernel.values()) / args.steps
        out["theta0_mode"] = {"kernel_ms_per_step": kern_ms, "other_ms_per_step": ms_step - kern_ms,
                              "note": "in-place: the other time is the host-to-device refill of theta0 "
                                      "(the paper hides it behind ordinary steps); host: theta0 is read "
                                      "by the kernels from pinned host memory"}
    if not args.no_e2e and args.theta0 == "device":
        need = 5 * 2 * w.numel
        avail = host_available_bytes() / max(1, world)
        ew = w
        if need > 0.5 * avail:
            ew = W.scaled(w, int(0.5 * avail / 10))
        del th, t0, sim, gs, go
        torch.cuda.empty_cache()
        e2e = e2e_run(ew, make_session, steps=max(2, min(args.steps, 5)), warmup=1, world=world)
        if out is not None:
            out["e2e"] = e2e
    if out is not None and not args.no_cpu_baseline and world == 1:
        # the oracle on every host core (one tensor per thread at a time), and
        # on one core as before
        cores = max(1, len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1))
        secs, b, n, sample = oracle_run(w, 40_000_000, threads=cores)
        secs1, b1, n1, sample1 = oracle_run(w, 10_000_000)
        out["cpu_baseline"] = {"value": b / secs / 1e9, "unit": UNIT, "cores": cores, "kind": "oracle",
                               "sample": f"{sample} (the single-threaded C++ oracle on {cores} threads, one "
                                         f"tensor each at a time; forward + gradient map, {secs:.1f} s wall)",
                               "params_per_s": n / secs,
                               "one_core": {"value": b1 / secs1 / 1e9, "unit": UNIT, "cores": 1,
                                            "sample": f"{sample1} ({secs1:.1f} s)", "params_per_s": n1 / secs1}}
    if out is not None:
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()
    return 0


SWEEP_LOG2N = (16, 18, 20, 22, 24, 26, 28, 30, 32)
SWEEP_KEEP = (0.1, 0.3, 0.5, 0.7, 0.9)
SWEEP_ALPHA = (1, 2)  # per tensor, per element
SWEEP_SIGMA = (0.0, 1e-4)


def run_sweep(args):
    """The flat-tensor sweep (one GPU): for each size and dtype the inputs are
    generated once; each (p_keep, alpha mode, sigma) point gets its own session."""
    from paper_2609_33437_gb300 import smat as S
    S.load_library()
    dev = torch.device("cuda")
    peak, peak_kind = measured_peaks()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)  # twice the L2
    stream = torch.cuda.current_stream()
    clocks = None if args.no_clocks else ClockSampler(torch.cuda.current_device())
    if clocks:
        clocks.mark()
    n_points, fracs = 0, []
    with open(args.sweep, "w") as out:
        for log2n in [x for x in SWEEP_LOG2N if args.sweep_min_log2n <= x <= args.sweep_max_log2n]:
            for dt in (W.F32, W.BF16):
                w0 = W.flat_sweep(log2n, dt, 0.5, 1, 0.0)
                th, t0, sim, gs, go = W.generate(w0, device=dev)
                b = 2 if dt == W.BF16 else 4
                n = 1 << log2n
                for keep in SWEEP_KEEP:
                    for am in SWEEP_ALPHA:
                        for sig in SWEEP_SIGMA:
                            w = W.flat_sweep(log2n, dt, keep, am, sig)
                            sess = S.SmatSession(th, t0, sim, [keep], [sig], [0.0], seed=w.seed,
                                                 alpha_min=w.alpha_min, alpha_max=w.alpha_max, alpha_mode=am,
                                                 noise=w.noise, draw_bits=args.draw_bits)

                            def fwd(s):
                                sess.simulate_multi(s)

                            def both(s):
                                sess.simulate_multi(s)
                                sess.swap()
                                sess.grad_map_multi(s, gs, go)
                                sess.swap()

                            rec = {"log2n": log2n, "dtype": "bf16" if dt == W.BF16 else "f32", "keep": keep,
                                   "alpha": "per-tensor" if am == 1 else "per-element", "sigma": sig}
                            for name, fn, nbytes in (("fwd", fwd, 3 * b * n), ("fwd_grad", both, 5 * b * n)):
                                times = []
                                for r in range(23):
                                    flush.zero_()
                                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                                    e0.record(stream)
                                    fn(r)
                                    e1.record(stream)
                                    e1.synchronize()
                                    if r >= 3:
                                        times.append(e0.elapsed_time(e1))
                                ms = statistics.median(times)
                                rec[name + "_ms"] = ms
                                rec[name + "_gbs"] = nbytes / (ms * 1e-3) / 1e9
                                rec[name + "_frac"] = rec[name + "_gbs"] / peak
                            sess.close()
                            out.write(json.dumps(rec) + "\n")
                            n_points += 2
                            if log2n >= 28:
                                fracs.append(rec["fwd_grad_frac"])
                del th, t0, sim, gs, go
                torch.cuda.empty_cache()
    if clocks:
        clocks.mark()
    clk = clocks.stop() if clocks else None
    print(json.dumps({"sweep": args.sweep, "points": n_points, "peak": peak, "peak_kind": peak_kind,
                      "median_fwd_grad_frac_n_ge_2^28": statistics.median(fracs) if fracs else None,
                      "clocks": clk, "l2": "256 MB written before every timed repetition"}))
    return 0


def run_schedule(args, d=4096, layers=8, tokens=8192, period=4, steps=32, warmup=4, rounds=3):
    """Training-loop overhead of the periodic schedule (Sec. 4.3: t = 4, one
    simulated-loss step per period) over plain fine-tuning, on a synthetic
    bf16 MLP stack (layers x [d -> 4d -> d] with residuals, about 1.07e9
    parameters) with fused AdamW (weight decay 1e-3) and random tokens: the
    paper's method settings (uniform Perturb, drop probability 0.5 on the
    matrices, global alpha ~ U[0.3, 1)). Three loops of `steps` steps each:
    plain, SMAT with theta0 in HBM, SMAT in-place with theta0 in pinned host
    memory (refilled on a side stream during the ordinary steps). The three
    loops run `rounds` times interleaved (clocks and power drift between
    runs); the median of each is reported, with the clocks seen."""
    from paper_2609_33437_gb300 import smat as S
    from paper_2609_33437_gb300.schedule import PeriodicSmat
    S.load_library()
    dev = torch.device("cuda")

    class Block(torch.nn.Module):
        def __init__(self):
            super().__init__()
            self.up = torch.nn.Linear(d, 4 * d)
            self.down = torch.nn.Linear(4 * d, d)

        def forward(self, x):
            return x + self.down(torch.nn.functional.gelu(self.up(x)))

    def build():
        torch.manual_seed(0)
        return torch.nn.Sequential(*[Block() for _ in range(layers)]).to(device=dev, dtype=torch.bfloat16)

    x = torch.randn(tokens, d, device=dev, dtype=torch.bfloat16)

    def run(mode):
        model = build()
        ps = list(model.parameters())
        opt = torch.optim.AdamW(ps, lr=1e-5, weight_decay=1e-3, fused=True)
        sched = None
        if mode != "ft":
            theta0 = [p.detach().clone() for p in ps]
            keeps = [0.5 if p.dim() == 2 else 1.0 for p in ps]
            kw = dict(seed=1, alpha_min=0.3, alpha_max=1.0, alpha_mode=S.SMAT_ALPHA_GLOBAL,
                      noise=S.SMAT_NOISE_UNIFORM, period=period)
            if mode == "smat":
                sched = PeriodicSmat(ps, keeps, [1e-4] * len(ps), theta0=theta0, **kw)
            else:
                sched = PeriodicSmat(ps, keeps, [1e-4] * len(ps), host_theta0=[t.cpu().pin_memory() for t in theta0],
                                     **kw)
                del theta0

        def one(step):
            if sched:
                sched.before_forward(step)
            model(x).float().square().mean().backward()
            if sched:
                sched.after_backward(step)
            opt.step()
            opt.zero_grad(set_to_none=False)

        for s in range(warmup):
            one(s)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for s in range(warmup, warmup + steps):
            one(s)
        if sched is not None and sched.refilled is not None:
            torch.cuda.current_stream().wait_event(sched.refilled)
        e1.record()
        torch.cuda.synchronize()
        n = sum(p.numel() for p in ps)
        if sched:
            sched.close()
        del model, opt, sched
        torch.cuda.empty_cache()
        return e0.elapsed_time(e1) / steps, n

    clocks = None if args.no_clocks else ClockSampler(torch.cuda.current_device())
    if clocks:
        clocks.mark()
    times = {"ft": [], "smat": [], "inplace": []}
    n = 0
    for _ in range(rounds):
        for mode in times:
            t, n = run(mode)
            times[mode].append(t)
    if clocks:
        clocks.mark()
    clk = clocks.stop() if clocks else None
    ft, smat, inpl = (statistics.median(times[m]) for m in ("ft", "smat", "inplace"))
    print(json.dumps({"schedule": "periodic SMAT, t = %d" % period, "params": n, "tokens_per_step": tokens,
                      "model": f"{layers} x MLP block d={d} (bf16, residual), fused AdamW",
                      "ft_ms_per_step": ft, "smat_ms_per_step": smat, "smat_inplace_ms_per_step": inpl,
                      "overhead_pct": 100.0 * (smat - ft) / ft, "overhead_inplace_pct": 100.0 * (inpl - ft) / ft,
                      "speed_vs_ft": ft / smat, "speed_vs_ft_inplace": ft / inpl,
                      "runs_ms_per_step": times, "steps": steps, "warmup": warmup, "clocks": clk}))
    return 0


def run_merge(args):
    """Merging K synthetic experts of the chosen list (theta_j = theta0 +
    delta_j, delta_j ~ N(0, delta_std^2) per the list's recipe) with the given
    method: gamma 0.3 (TA, DARE, TIES), DARE drop 0.3, TIES retention 0.5 (the
    paper's calibrated settings, App. B). Algorithmic bytes per element: the
    merge reads theta0 and the K experts and writes the result, (K + 2) b; TIES
    adds three radix-select passes that each read theta0 and every expert,
    3 (K + 1) b: (4 K + 5) b in all."""
    from paper_2609_33437_gb300 import smat as S
    S.load_library()
    dev = torch.device("cuda")
    w = workload(args)
    K = args.experts
    method = {"wa": S.SMAT_MERGE_WA, "ta": S.SMAT_MERGE_TA, "dare": S.SMAT_MERGE_DARE_TA, "ties": S.SMAT_MERGE_TIES}[args.merge]
    tdt = W.torch_dtype(w.dtype)
    t0s, exs, outs = [], [], []
    for k, spec in enumerate(w.tensors):
        g = torch.Generator(device=dev).manual_seed(w.data_seed * 100003 + k)
        t0 = torch.randn(spec.numel, generator=g, device=dev) * w.theta0_std
        ex = [(t0 + torch.randn(spec.numel, generator=g, device=dev) * w.delta_std).to(tdt) for _ in range(K)]
        t0s.append(t0.to(tdt))
        exs.append(ex)
        outs.append(torch.empty(spec.numel, dtype=tdt, device=dev))
        del t0
    kw = dict(gamma=0.3, p_drop=0.3, retention=0.5, seed=1)
    for _ in range(max(1, args.warmup)):
        S.merge(t0s, exs, outs, method, **kw)
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        S.merge(t0s, exs, outs, method, **kw)
        e1.record()
        e1.synchronize()
        times.append(e0.elapsed_time(e1))
    ms = statistics.median(times)
    b = 2 if w.dtype == W.BF16 else 4
    nbytes = (K + 2) * b * w.numel + (3 * (K + 1) * b * w.numel if method == S.SMAT_MERGE_TIES else 0)
    peak, peak_kind = measured_peaks()
    print(json.dumps({"merge": args.merge, "experts": K, "workload": w.name, "elements": w.numel,
                      "ms": ms, "gbs": nbytes / (ms * 1e-3) / 1e9, "frac_of_measured_peak": nbytes / (ms * 1e-3) / 1e9 / peak,
                      "algorithmic_bytes": nbytes, "runs_ms": times, "settings": kw}))
    return 0


def run_adamw(args):
    """The gradient map fused with an AdamW step (smat_grad_map_adamw_multi)
    on the chosen list, beside the plain gradient map into a separate buffer.
    Each timed call follows a forward of its own SMAT step (new mask), as in
    training; the moments start warm (m1 ~ N(0, 1e-6), m2 ~ U[0, 1e-6), as
    after earlier optimizer steps). A second series times the first optimizer
    step, from zero moments (reset outside the timed region) on one mask.
    Algorithmic bytes per element of the fused call: read g~, theta, m1, m2
    and write theta, m1, m2, g + 2 b + 16 (22 for bf16 gradients and
    parameters); the plain map moves 2 g, and an update after it would move
    g + 2 b + 16 again (26 in all). Inputs are larger than L2, so no flush
    between calls."""
    from paper_2609_33437_gb300 import smat as S
    S.load_library()
    dev = torch.device("cuda")
    w = workload(args)
    th, t0, sim, gs, go = W.generate(w, device=dev)
    gen = torch.Generator(device=dev).manual_seed(w.data_seed + 17)
    m1 = [torch.randn(t.numel, generator=gen, device=dev) * 1e-3 for t in w.tensors]
    m2 = [torch.rand(t.numel, generator=gen, device=dev) * 1e-6 for t in w.tensors]
    sess = S.SmatSession(th, t0, sim, [t.keep_prob for t in w.tensors], [t.sigma for t in w.tensors],
                         [t.sigma_rel for t in w.tensors], seed=w.seed, alpha_min=w.alpha_min,
                         alpha_max=w.alpha_max, alpha_mode=w.alpha_mode, noise=w.noise,
                         philox_rounds=args.philox_rounds, draw_bits=args.draw_bits)
    hp = dict(lr=1e-5, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.01)

    def ev():
        return torch.cuda.Event(enable_timing=True)

    fused, plain = [], []
    n_iter = max(3, args.warmup) + args.steps
    for i in range(n_iter):
        sess.simulate_multi(i)
        e = [ev() for _ in range(4)]
        e[0].record()
        sess.grad_map_adamw_multi(i, gs, m1, m2, adam_step=i + 1, **hp)
        e[1].record()
        e[2].record()
        sess.grad_map_multi(i, gs, go)
        e[3].record()
        e[3].synchronize()
        if i >= n_iter - args.steps:
            fused.append(e[0].elapsed_time(e[1]))
            plain.append(e[2].elapsed_time(e[3]))
    cold = []
    for i in range(max(3, args.warmup) + args.steps):
        for x in m1 + m2:
            x.zero_()
        e = [ev() for _ in range(2)]
        e[0].record()
        sess.grad_map_adamw_multi(n_iter - 1, gs, m1, m2, adam_step=1, **hp)
        e[1].record()
        e[1].synchronize()
        if i >= max(3, args.warmup):
            cold.append(e[0].elapsed_time(e[1]))
    n = w.numel
    gb = 2 if w.gdtype == W.BF16 else 4
    pb = 2 if w.dtype == W.BF16 else 4
    fused_bytes = (gb + 2 * pb + 16) * n
    map_bytes = 2 * gb * n
    ms_f, ms_m, ms_c = statistics.median(fused), statistics.median(plain), statistics.median(cold)
    peak, peak_kind = measured_peaks()
    gbs = fused_bytes / (ms_f * 1e-3) / 1e9
    rec = recorded_traffic("gradmap_adamw", w.name)
    assert sess.poll_errors() == 0
    print(json.dumps({"adamw": True, "workload": w.name, "elements": n, "fused_ms": ms_f,
                      "fused_gbs": gbs, "fused_frac": gbs / peak, "peak_gbs": peak, "peak_kind": peak_kind,
                      "fused_bytes_per_elem": fused_bytes / n, "first_step_ms": ms_c,
                      "first_step_gbs": fused_bytes / (ms_c * 1e-3) / 1e9, "grad_map_ms": ms_m,
                      "grad_map_gbs": map_bytes / (ms_m * 1e-3) / 1e9,
                      "separate_bytes_per_elem": 3 * gb + 2 * pb + 16,
                      "traffic": rec["dram_bytes_per_launch"] if rec else None,
                      "runs_ms": {"fused": fused, "first_step": cold, "grad_map": plain}, "hyper": hp,
                      "draw_bits": args.draw_bits, "philox_rounds": args.philox_rounds}))
    sess.close()
    return 0


def main():
    args = parse()
    if args.merge:
        return run_merge(args)
    if args.adamw:
        return run_adamw(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    if args.schedule:
        return run_schedule(args)
    return run_smat(args)


if __name__ == "__main__":
    sys.exit(main())
