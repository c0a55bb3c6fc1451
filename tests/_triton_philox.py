"""Evaluate Philox-4x32-R blocks with Triton's own Philox (run on the CPU by
Triton's interpreter). Used as an independent library pin of the oracle's
Philox block; run as a subprocess so TRITON_INTERPRET is set before import.

stdin: JSON {"ctr": [[c0,c1,c2,c3],...], "seed": [s,...], "rounds": R}
stdout: JSON [[w0,w1,w2,w3], ...]
"""
import json
import os
import sys

os.environ["TRITON_INTERPRET"] = "1"

import torch  # noqa: E402
import triton  # noqa: E402
import triton.language as tl  # noqa: E402


@triton.jit
def _philox_kernel(c_ptr, seed_lo_ptr, seed_hi_ptr, out_ptr, N: tl.constexpr, R: tl.constexpr):
    i = tl.arange(0, N)
    c0 = tl.load(c_ptr + 4 * i + 0)
    c1 = tl.load(c_ptr + 4 * i + 1)
    c2 = tl.load(c_ptr + 4 * i + 2)
    c3 = tl.load(c_ptr + 4 * i + 3)
    k0 = tl.load(seed_lo_ptr + i).to(tl.uint32, bitcast=True)
    k1 = tl.load(seed_hi_ptr + i).to(tl.uint32, bitcast=True)
    a, b, c, d = tl.random.philox_impl(c0.to(tl.uint32, bitcast=True), c1.to(tl.uint32, bitcast=True),
                                       c2.to(tl.uint32, bitcast=True), c3.to(tl.uint32, bitcast=True),
                                       k0, k1, R)
    tl.store(out_ptr + 4 * i + 0, a.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 1, b.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 2, c.to(tl.int32, bitcast=True))
    tl.store(out_ptr + 4 * i + 3, d.to(tl.int32, bitcast=True))


def main():
    req = json.load(sys.stdin)
    ctr = req["ctr"]
    n = len(ctr)
    N = 1
    while N < n:
        N *= 2

    def i32(v):
        v &= 0xFFFFFFFF
        return v - (1 << 32) if v >= (1 << 31) else v

    c = torch.zeros(4 * N, dtype=torch.int32)
    lo = torch.zeros(N, dtype=torch.int32)
    hi = torch.zeros(N, dtype=torch.int32)
    for k in range(n):
        for w in range(4):
            c[4 * k + w] = i32(ctr[k][w])
        lo[k] = i32(req["seed"][k] & 0xFFFFFFFF)
        hi[k] = i32(req["seed"][k] >> 32)
    out = torch.zeros(4 * N, dtype=torch.int32)
    _philox_kernel[(1,)](c, lo, hi, out, N=N, R=req["rounds"])
    res = [[int(out[4 * k + w]) & 0xFFFFFFFF for w in range(4)] for k in range(n)]
    json.dump(res, sys.stdout)


if __name__ == "__main__":
    main()
