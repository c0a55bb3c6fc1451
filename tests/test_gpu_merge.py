"""Merge kernels (the evaluation side, Eq. merged-state): WA, TA, DARE + TA and
TIES over K experts, bit-identical to the CPU oracle on ragged lists (vector
and element paths), including the TIES trim thresholds, in place, with DARE
ties and element offsets, and on inputs with many equal magnitudes."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_33437_gb300 import smat as S

from _parity import f32_of, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


METHODS = {S.SMAT_MERGE_WA: O.MERGE_WA, S.SMAT_MERGE_TA: O.MERGE_TA, S.SMAT_MERGE_DARE_TA: O.MERGE_DARE_TA,
           S.SMAT_MERGE_TIES: O.MERGE_TIES}


def _experts(sizes, K, dtype, seed, quantum=None):
    g = torch.Generator(device="cuda").manual_seed(seed)
    tdt = torch.bfloat16 if dtype == O.BF16 else torch.float32
    t0s, exs = [], []
    for n in sizes:
        t0 = torch.randn(n, device="cuda", generator=g) * 0.02
        ex = []
        for _ in range(K):
            d = torch.randn(n, device="cuda", generator=g) * 1e-3
            if quantum:
                d = torch.round(d / quantum) * quantum
            ex.append((t0 + d).to(tdt))
        t0s.append(t0.to(tdt))
        exs.append(ex)
    return t0s, exs


def _check(t0s, exs, outs, dtype, method, kw, elem_offsets=None, thr=None):
    K = len(exs[0])
    for k, (t0, ex, out) in enumerate(zip(t0s, exs, outs)):
        ref, rthr = O.merge(METHODS[method], to_host(t0), [to_host(x) for x in ex], dtype=dtype,
                            gamma=kw.get("gamma", 1.0), p_drop=kw.get("p_drop", 0.0),
                            retention=kw.get("retention", 1.0), seed=kw.get("seed", 0), tensor_id=k,
                            elem_offset=0 if elem_offsets is None else elem_offsets[k])
        got = to_host(out)
        view = np.uint16 if dtype == O.BF16 else np.uint32
        assert np.array_equal(got.view(view), ref.view(view)), f"tensor {k}"
        if thr is not None:
            assert np.array_equal(thr[k].cpu().numpy().view(np.uint32), rthr), f"tensor {k} thresholds"


SIZES = [1, 15, 16, 17, 4096, 65_536 + 33, 131_073]


@pytest.mark.parametrize("method", list(METHODS))
@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_merge_matches_oracle(method, dtype):
    K = 5
    t0s, exs = _experts(SIZES, K, dtype, seed=100 + method)
    outs = [torch.empty_like(t) for t in t0s]
    kw = dict(gamma=0.7, p_drop=0.3, retention=0.3, seed=99)  # p_drop 0.3: threshold with low bits (ties)
    thr = S.merge(t0s, exs, outs, method, return_thresholds=method == S.SMAT_MERGE_TIES, **kw)
    torch.cuda.synchronize()
    _check(t0s, exs, outs, dtype, method, kw, thr=thr)


@pytest.mark.parametrize("method", list(METHODS))
def test_merge_in_place_equals_out_of_place(method):
    t0s, exs = _experts([70_001, 4096 + 5], 3, O.BF16, seed=7)
    kw = dict(gamma=0.5, p_drop=0.5, retention=0.5, seed=3)
    outs = [torch.empty_like(t) for t in t0s]
    S.merge(t0s, exs, outs, method, **kw)
    inplace = [t.clone() for t in t0s]
    S.merge(inplace, exs, inplace, method, **kw)
    torch.cuda.synchronize()
    for a, b in zip(outs, inplace):
        assert torch.equal(a.view(torch.int16), b.view(torch.int16))


@pytest.mark.parametrize("method", [S.SMAT_MERGE_DARE_TA, S.SMAT_MERGE_TIES])
def test_merge_element_path_and_offsets(method):
    """Unaligned pointers take the element path; elem_offset keys the DARE
    masks like a shard of a larger tensor."""
    n, K = 33_333, 4
    t0s, exs = _experts([n + 3], K, O.F32, seed=11)
    base, ex_base = t0s[0], exs[0]
    t0 = base[3:]
    ex = [x[3:] for x in ex_base]  # 12-byte offset: not 32-byte aligned
    out = torch.empty(n + 8, device="cuda")[5:5 + n]
    kw = dict(gamma=1.0, p_drop=0.3, retention=0.5, seed=5)
    S.merge([t0], [ex], [out], method, elem_offsets=[1000], **kw)
    torch.cuda.synchronize()
    _check([t0], [ex], [out], O.F32, method, kw, elem_offsets=[1000])


def test_merge_ties_many_equal_magnitudes():
    """Deltas on a coarse grid: thousands of equal |Delta| at the threshold,
    all kept, thresholds equal to the oracle's."""
    t0s, exs = _experts([100_003, 5000], 6, O.F32, seed=13, quantum=5e-4)
    outs = [torch.empty_like(t) for t in t0s]
    kw = dict(gamma=1.0, retention=0.2)
    thr = S.merge(t0s, exs, outs, S.SMAT_MERGE_TIES, return_thresholds=True, **kw)
    torch.cuda.synchronize()
    _check(t0s, exs, outs, O.F32, S.SMAT_MERGE_TIES, kw, thr=thr)


def test_merge_argument_errors():
    t0s, exs = _experts([1000], 2, O.F32, seed=1)
    out = [torch.empty_like(t0s[0])]
    for bad in (dict(p_drop=1.0), dict(retention=0.0), dict(gamma=float("inf")), dict(philox_rounds=8)):
        with pytest.raises(S.SmatError):
            S.merge(t0s, exs, out, S.SMAT_MERGE_DARE_TA, **bad)
    with pytest.raises(S.SmatError):
        S.merge(t0s, [exs[0] * 9], out, S.SMAT_MERGE_TA)  # 18 experts > 16
    with pytest.raises(S.SmatError):
        S.merge(t0s, exs, [exs[0][0]], S.SMAT_MERGE_TA)  # out is an expert
    with pytest.raises(S.SmatError):
        S.merge(t0s + [t0s[0].to(torch.bfloat16)], exs + [[x.to(torch.bfloat16) for x in exs[0]]],
                out + [torch.empty(1000, device="cuda", dtype=torch.bfloat16)], S.SMAT_MERGE_TA)  # two dtypes


def test_merge_dare_seven_rounds():
    """DARE masks with the 7-round stream option equal the oracle's."""
    t0s, exs = _experts([70_001, 4096], 3, O.BF16, seed=17)
    outs = [torch.empty_like(t) for t in t0s]
    S.merge(t0s, exs, outs, S.SMAT_MERGE_DARE_TA, gamma=0.5, p_drop=0.3, seed=8, philox_rounds=7)
    torch.cuda.synchronize()
    for k, (t0, ex, out) in enumerate(zip(t0s, exs, outs)):
        ref, _ = O.merge(O.MERGE_DARE_TA, to_host(t0), [to_host(x) for x in ex], dtype=O.BF16, gamma=0.5,
                         p_drop=0.3, seed=8, tensor_id=k, rounds=7)
        assert np.array_equal(to_host(out).view(np.uint16), ref.view(np.uint16)), k


@pytest.mark.parametrize("K", [1, 2, 8, 9, 15, 16])
def test_merge_dare_expert_counts(K):
    """DARE with one to sixteen experts (the kernel loads experts in batches
    of four, so every remainder occurs) equals the oracle."""
    t0s, exs = _experts([17, 4096, 65_536 + 33], K, O.BF16, seed=40 + K)
    outs = [torch.empty_like(t) for t in t0s]
    kw = dict(gamma=0.6, p_drop=0.3, seed=5)
    S.merge(t0s, exs, outs, S.SMAT_MERGE_DARE_TA, **kw)
    torch.cuda.synchronize()
    _check(t0s, exs, outs, O.BF16, S.SMAT_MERGE_DARE_TA, kw)


@pytest.mark.parametrize("method", list(METHODS))
@pytest.mark.parametrize("dtype", [O.F32, O.BF16])
def test_merge_special_values(method, dtype):
    """Signed zeros, infinities, NaN, subnormals and experts equal to theta0
    sprinkled into theta0 and the experts: every result equals the oracle's
    bit for bit, NaN matching any NaN (payloads differ between host and GPU).
    Retention keeps the TIES thresholds among the finite keys."""
    n, K = 20_000 + 7, 5
    g = torch.Generator().manual_seed(23)
    t0 = torch.randn(n, generator=g) * 0.02
    ex = [t0 + torch.randn(n, generator=g) * 1e-3 for _ in range(K)]
    specials = torch.tensor([0.0, -0.0, float("inf"), float("-inf"), float("nan"), 1e-40, -1e-40, 3e-39])
    for arr in [t0] + ex:
        pos = torch.randint(0, n, (n // 50,), generator=g)
        arr[pos] = specials[torch.randint(0, len(specials), (len(pos),), generator=g)]
    for e in range(K):  # Delta exactly 0 on a few coordinates
        pos = torch.randint(0, n, (n // 100,), generator=g)
        ex[e][pos] = t0[pos]
    tdt = torch.bfloat16 if dtype == O.BF16 else torch.float32
    t0d = t0.to(tdt).cuda()
    exd = [x.to(tdt).cuda() for x in ex]
    out = torch.empty_like(t0d)
    kw = dict(gamma=0.7, p_drop=0.3, retention=0.3, seed=4)
    S.merge([t0d], [exd], [out], method, **kw)
    torch.cuda.synchronize()
    ref, _ = O.merge(METHODS[method], to_host(t0d), [to_host(x) for x in exd], dtype=dtype, tensor_id=0, **kw)
    got = to_host(out)
    gf, rf = f32_of(got), f32_of(ref)
    view = np.uint16 if dtype == O.BF16 else np.uint32
    nan_g, nan_r = np.isnan(gf), np.isnan(rf)
    assert np.array_equal(nan_g, nan_r)
    assert np.array_equal(got.view(view)[~nan_g], ref.view(view)[~nan_r])
